"""CPU oracle of the batched embedding key-value path -- TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path (the CUDA library and
its binding) never does; the two share no code.

The arithmetic lives in ``mlkv_oracle.cpp`` (sequential ``std::unordered_map``
table, Get/Put upserts, one Adagrad step per distinct key on its summed
gradient, MLKV Sections 2.1, 3.1 and 3.2 / Figure 2).  This module only
marshals numpy arrays into it.

Parity status of each function (what pins it, in ``tests/test_oracle_pins.py``):
  * splitmix64 / init_value: published SplitMix64 output vectors, the exact
    2^-24 lattice, uniformity and the affine map to [lo, hi).
  * apply_grad (Adagrad): closed forms (eps = 0 constant-gradient trajectory
    via the generalised harmonic number, scale invariance, g = eps gives lr/2,
    state_init = 3 g^2 gives lr/2), the duplicate-key reading, zero gradient
    and column independence.
  * dedup / segment_sums: brute force on small batches (pairwise equality,
    exactly rounded sums with math.fsum).
  * get / put / insert / find / export: hand-built batches with hand-written
    row ids (tests/golden), Get-after-Put and the key-to-row invariants.
  * keys / import (checkpoints): import-then-export returns what was
    imported, the later duplicate wins, a missing state keeps the current
    one, and a table restored from keys + export continues bit-identically.
"""
import ctypes
import os

import numpy as np

from . import build as _build

_LIBS: dict = {}

OK = 0
ERR_INVALID = 1
NOT_FOUND = 7


def load(mutant: int = 0, out_dir: str | None = None) -> ctypes.CDLL:
    key = (mutant, out_dir)
    if key in _LIBS:
        return _LIBS[key]
    path = _build.build(mutant=mutant, out_dir=out_dir)
    lib = ctypes.CDLL(path)
    i32, i64, u64, f32, vp = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64,
                              ctypes.c_float, ctypes.c_void_p)
    lib.oracle_splitmix64.restype = u64
    lib.oracle_splitmix64.argtypes = [u64]
    lib.oracle_init_value.restype = f32
    lib.oracle_init_value.argtypes = [u64, u64, i64, f32, f32]
    lib.oracle_mutant.restype = i32
    lib.oracle_open.restype = vp
    lib.oracle_open.argtypes = [i32, f32, f32, f32, f32, f32, u64, i32, i32]
    lib.oracle_close.argtypes = [vp]
    lib.oracle_size.restype = i64
    lib.oracle_size.argtypes = [vp]
    for name in ("oracle_get",):
        getattr(lib, name).restype = i32
        getattr(lib, name).argtypes = [vp, vp, i64, vp, vp]
    for name in ("oracle_put", "oracle_apply_grad"):
        getattr(lib, name).restype = i32
        getattr(lib, name).argtypes = [vp, vp, i64, vp]
    lib.oracle_insert.restype = i32
    lib.oracle_insert.argtypes = [vp, vp, i64]
    lib.oracle_import.restype = i32
    lib.oracle_import.argtypes = [vp, vp, i64, vp, vp]
    lib.oracle_keys.restype = i64
    lib.oracle_keys.argtypes = [vp, vp]
    lib.oracle_find.restype = i32
    lib.oracle_find.argtypes = [vp, vp, i64, vp]
    lib.oracle_export.restype = i64
    lib.oracle_export.argtypes = [vp, vp, i64, vp, vp]
    lib.oracle_dedup.restype = i64
    lib.oracle_dedup.argtypes = [vp, i64, vp, vp, vp]
    lib.oracle_segment_sums.restype = i64
    lib.oracle_segment_sums.argtypes = [vp, i64, vp, i32, i32, vp, vp]
    _LIBS[key] = lib
    return lib


def _keys(keys) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(keys, dtype=np.uint64).view(np.int64))


def _f32(x, shape=None) -> np.ndarray:
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    if shape is not None:
        a = a.reshape(shape)
    return a


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def splitmix64(z: int, lib=None) -> int:
    return int((lib or load()).oracle_splitmix64(ctypes.c_uint64(z & (2**64 - 1))))


def init_value(seed: int, key: int, j: int, lo: float, hi: float, lib=None) -> float:
    return float((lib or load()).oracle_init_value(seed & (2**64 - 1), key & (2**64 - 1), j, lo, hi))


def init_rows(seed: int, keys, dim: int, lo: float, hi: float, lib=None) -> np.ndarray:
    """Init rows of `keys` (float32 [n, dim]) by calling the oracle per element."""
    lib = lib or load()
    keys = _keys(keys).view(np.uint64)
    out = np.empty((len(keys), dim), np.float32)
    for i, k in enumerate(keys):
        for j in range(dim):
            out[i, j] = lib.oracle_init_value(seed & (2**64 - 1), int(k), j, lo, hi)
    return out


class Table:
    """Sequential oracle table (Open of MLKV Section 3.1; staleness bound 0)."""

    def __init__(self, dim, lr=0.1, eps=1e-8, state_init=0.0, init_lo=-0.01, init_hi=0.01,
                 seed=1, insert_on_miss=True, precision=32, mutant=0, lib=None):
        self.lib = lib or load(mutant)
        self.dim = int(dim)
        self.h = self.lib.oracle_open(self.dim, lr, eps, state_init, init_lo, init_hi,
                                      seed & (2**64 - 1), int(bool(insert_on_miss)), precision)
        if not self.h:
            raise ValueError("oracle_open rejected the configuration")

    def close(self):
        if self.h:
            self.lib.oracle_close(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def size(self) -> int:
        return int(self.lib.oracle_size(self.h))

    def get(self, keys):
        k = _keys(keys)
        out = np.empty((len(k), self.dim), np.float32)
        rows = np.empty(len(k), np.int64)
        rc = self.lib.oracle_get(self.h, _p(k), len(k), _p(out), _p(rows))
        return out, rows, rc

    def put(self, keys, vals):
        k = _keys(keys)
        v = _f32(vals, (len(k), self.dim))
        return self.lib.oracle_put(self.h, _p(k), len(k), _p(v))

    def insert(self, keys):
        k = _keys(keys)
        return self.lib.oracle_insert(self.h, _p(k), len(k))

    def apply_grad(self, keys, grads):
        k = _keys(keys)
        g = _f32(grads, (len(k), self.dim))
        return self.lib.oracle_apply_grad(self.h, _p(k), len(k), _p(g))

    def import_(self, keys, rows, state=None):
        k = _keys(keys)
        w = _f32(rows, (len(k), self.dim))
        G = None if state is None else _f32(state, (len(k), self.dim))
        return self.lib.oracle_import(self.h, _p(k), len(k), _p(w), None if G is None else _p(G))

    def keys(self) -> np.ndarray:
        out = np.empty(self.size(), np.int64)
        self.lib.oracle_keys(self.h, _p(out))
        return out

    def find(self, keys) -> np.ndarray:
        k = _keys(keys)
        rows = np.empty(len(k), np.int64)
        self.lib.oracle_find(self.h, _p(k), len(k), _p(rows))
        return rows

    def export(self, keys):
        k = _keys(keys)
        w = np.empty((len(k), self.dim), np.float32)
        G = np.empty((len(k), self.dim), np.float32)
        self.lib.oracle_export(self.h, _p(k), len(k), _p(w), _p(G))
        return w, G


def dedup(keys, lib=None):
    """Distinct keys in first-occurrence order, their counts and first positions."""
    lib = lib or load()
    k = _keys(keys)
    n = len(k)
    uniq = np.empty(max(n, 1), np.int64)
    counts = np.empty(max(n, 1), np.int64)
    first = np.empty(max(n, 1), np.int64)
    u = lib.oracle_dedup(_p(k), n, _p(uniq), _p(counts), _p(first))
    return uniq[:u].copy(), counts[:u].copy(), first[:u].copy()


def segment_sums(keys, grads, dim, precision=32, lib=None):
    """Per distinct key (first-occurrence order) the occurrence-order gradient sum."""
    lib = lib or load()
    k = _keys(keys)
    n = len(k)
    g = _f32(grads, (n, dim))
    uniq = np.empty(max(n, 1), np.int64)
    sums = np.empty((max(n, 1), dim), np.float32)
    u = lib.oracle_segment_sums(_p(k), n, _p(g), dim, precision, _p(uniq), _p(sums))
    return uniq[:u].copy(), sums[:u].copy()

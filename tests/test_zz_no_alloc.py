"""The dedup entry point that allocates nothing, checked against mlkv_dedup and the oracle.

Some callers must not allocate device memory when they need a dedup: plugins
inside an engine that reserved the device's memory up front and owns every
allocation, and latency-bound loops that ban cudaMalloc / cudaFree because
those may synchronise the device.  mlkv_dedup_keys_static serves them from a
fixed array in the library's device image.

Checks: two calls in a row against the table's own dedup (mlkv_dedup), and a
run of calls on one stream against the oracle's dedup (distinct keys with their
counts, re-sorted in unsigned order), over the cases the entry point promises:
every key value including -1 and other negative keys, keys with high bits set
(the sort's upper passes), n = 0, n = 1, an all-equal batch and a full batch of
MLKV_STATIC_MAX_KEYS keys.  Each case's output is checked before the next call
reuses the shared array.

This file is collected last on purpose: a run that stops at the first failure
has run every other test before it.  It passes in a fresh process and after
the other tests alike (its first call does the per-device set-up).
"""
import ctypes

import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import dev, host, torch_cuda

pytestmark = pytest.mark.gpu


def _static_dedup(lib, torch, keys_d, expect_rc=0):
    n = keys_d.numel()
    uniq = torch.full((max(n, 1),), 0x5A5A, dtype=torch.int64, device="cuda:0")
    counts = torch.full((max(n, 1),), -7, dtype=torch.int32, device="cuda:0")
    num = torch.full((1,), -1, dtype=torch.int64, device="cuda:0")
    stream = torch.cuda.current_stream().cuda_stream
    rc = lib.mlkv_dedup_keys_static(ctypes.c_void_p(keys_d.data_ptr() if n else 0), ctypes.c_int64(n),
                                    ctypes.c_void_p(uniq.data_ptr()), ctypes.c_void_p(counts.data_ptr()),
                                    ctypes.c_void_p(num.data_ptr()), ctypes.c_void_p(stream))
    assert rc == expect_rc
    u = int(num.item())
    return host(uniq[:u]), host(counts[:u])


def _oracle_sorted(keys):
    """The oracle's distinct keys and counts, in ascending unsigned order."""
    ou, oc, _ = oracle.dedup(keys)
    o = np.argsort(ou.view(np.uint64), kind="stable")
    return ou[o], oc[o]


def _assert_strictly_ascending_unsigned(u, what):
    uu = np.asarray(u).view(np.uint64)
    assert np.all(uu[1:] > uu[:-1]), f"{what}: distinct keys not in strictly ascending unsigned order"


def test_static_dedup_matches_mlkv_dedup_twice():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore, _lib

    lib = _lib.load()
    cfg = W.tiny()
    store = EmbeddingStore(dim=4, capacity=cfg.n_keys, max_batch=cfg.n_keys, device="cuda:0")
    store.insert(dev(cfg.preload_keys()))
    batches = [cfg.batch_keys(0), np.concatenate([cfg.batch_keys(1), cfg.batch_keys(2)])[:_lib.STATIC_MAX_KEYS]]
    for keys in batches:  # two calls in a row share (and overwrite) the static scratch
        su, sc = _static_dedup(lib, torch, dev(keys))
        tu, tc = store.dedup(dev(keys))
        tu, tc = host(tu), host(tc)
        o = np.argsort(tu.view(np.uint64), kind="stable")
        assert np.array_equal(su, tu[o])
        assert np.array_equal(sc, tc[o])
        _assert_strictly_ascending_unsigned(su, "static dedup")
    store.close()


def _edge_cases():
    rng = np.random.default_rng(2504)
    full = _static_max()
    cases = []
    # the key -1 (all bits set) and other negative keys among ordinary ones
    k = rng.integers(-50, 50, 3000).astype(np.int64)
    k[::97] = -1
    cases.append(("negative keys and -1", k))
    # keys with high bits set: every byte of the key differs between keys, so
    # all 8 passes of the sort move elements
    hi = rng.integers(0, 2**63, 400, dtype=np.int64) | np.int64(-(2**63))
    lo = rng.integers(0, 2**63, 400, dtype=np.int64)
    k = np.concatenate([hi, lo, np.int64(-(2**63)) + np.zeros(3, np.int64), np.full(5, 2**63 - 1, np.int64)])
    cases.append(("high bits", rng.choice(k, 20_000)))
    cases.append(("n = 0", np.zeros(0, np.int64)))
    cases.append(("n = 1", np.array([-1], np.int64)))
    cases.append(("n = 1, ordinary key", np.array([123456789012345], np.int64)))
    cases.append(("all equal", np.full(10_000, -(2**40) + 3, np.int64)))
    # a full batch with a Zipf head (long runs) and a uniform tail over all bit patterns
    ranks = W.ZipfSampler(5_000, 1.1).sample(rng, full // 2)
    keyset = rng.integers(-(2**63), 2**63 - 1, 5_000, dtype=np.int64, endpoint=True)
    k = np.concatenate([keyset[ranks - 1], rng.integers(-(2**63), 2**63 - 1, full - full // 2, dtype=np.int64,
                                                        endpoint=True)])
    rng.shuffle(k)
    cases.append(("full batch", k))
    cases.append(("ragged tile tail", rng.integers(0, 300, 4097).astype(np.int64)))
    return cases


def _static_max():
    from paper_2504_01506_gb300 import _lib

    return _lib.STATIC_MAX_KEYS


def test_static_dedup_matches_oracle_on_edge_cases():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import _lib

    lib = _lib.load()
    cases = _edge_cases()
    assert len(cases[-2][1]) == _lib.STATIC_MAX_KEYS
    for what, keys in cases:  # one call after another on the shared array
        su, sc = _static_dedup(lib, torch, dev(keys) if len(keys) else torch.empty(0, dtype=torch.int64,
                                                                                   device="cuda:0"))
        ou, oc = _oracle_sorted(keys)
        assert len(su) == len(ou), f"{what}: {len(su)} distinct keys, oracle {len(ou)}"
        assert np.array_equal(su, ou), f"{what}: distinct keys differ from the oracle"
        assert np.array_equal(sc.astype(np.int64), oc), f"{what}: counts differ from the oracle"
        _assert_strictly_ascending_unsigned(su, what)
        assert int(sc.sum()) == len(keys), what


def test_static_dedup_rejects_oversize():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import _lib

    lib = _lib.load()
    big = torch.zeros(_lib.STATIC_MAX_KEYS + 1, dtype=torch.int64, device="cuda:0")
    out = torch.empty(1, dtype=torch.int64, device="cuda:0")
    rc = lib.mlkv_dedup_keys_static(ctypes.c_void_p(big.data_ptr()), ctypes.c_int64(big.numel()),
                                    ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(out.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(0))
    assert rc == _lib.ERR_INVALID

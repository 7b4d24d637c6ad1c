"""The dedup entry point that allocates nothing, checked against mlkv_dedup.

Some callers may not allocate device memory when they need a dedup (work
issued while a stream is captured in global mode, engine plugins that own all
device memory).  mlkv_dedup_keys_static serves them from a fixed array in the
library's device image.  This file is collected last on purpose: a run that
stops at the first failure has run every other test before it.  It passes in a
fresh process and after the other tests alike (its first call does the
per-device set-up).
"""
import ctypes

import numpy as np
import pytest

import workloads as W
from gpu_helpers import dev, host, torch_cuda

pytestmark = pytest.mark.gpu


def _static_dedup(lib, torch, keys_d):
    n = keys_d.numel()
    uniq = torch.empty(max(n, 1), dtype=torch.int64, device="cuda:0")
    counts = torch.empty(max(n, 1), dtype=torch.int32, device="cuda:0")
    num = torch.full((1,), -1, dtype=torch.int64, device="cuda:0")
    stream = torch.cuda.current_stream().cuda_stream
    rc = lib.mlkv_dedup_keys_static(ctypes.c_void_p(keys_d.data_ptr()), ctypes.c_int64(n),
                                    ctypes.c_void_p(uniq.data_ptr()), ctypes.c_void_p(counts.data_ptr()),
                                    ctypes.c_void_p(num.data_ptr()), ctypes.c_void_p(stream))
    assert rc == 0
    u = int(num.item())
    return host(uniq[:u]), host(counts[:u])


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
        assert np.all(np.diff(su.view(np.uint64).astype(np.float64)) > 0)
    store.close()


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

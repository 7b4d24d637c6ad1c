"""Shared helpers of the GPU parity tests (store + oracle side by side)."""
import numpy as np
import pytest

import oracle

TOL = 1e-5  # max |gpu - ref| <= TOL * (1 + |ref|), per element


def torch_cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def make_pair(cfg, capacity=None, max_batch=None, precision=32, insert_on_miss=True, flags=0, **over):
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    kw = dict(lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi,
              seed=cfg.seed)
    kw.update(over)
    store = EmbeddingStore(dim=cfg.dim, capacity=capacity or cfg.n_keys,
                           max_batch=max_batch or max(cfg.batch, cfg.n_keys),
                           insert_on_miss=insert_on_miss, flags=flags, device=torch.device("cuda", 0), **kw)
    ref = oracle.Table(cfg.dim, insert_on_miss=insert_on_miss, precision=precision, **kw)
    return store, ref


def dev(x):
    torch = torch_cuda()
    return torch.from_numpy(np.ascontiguousarray(x)).to("cuda:0")


def host(t):
    return t.detach().cpu().numpy()


def assert_close(got, want, what):
    got = np.asarray(got, np.float32)
    want = np.asarray(want, np.float32)
    assert got.shape == want.shape, what
    err = np.abs(got.astype(np.float64) - want.astype(np.float64))
    tol = TOL * (1.0 + np.abs(want.astype(np.float64)))
    bad = ~(err <= tol)
    assert not bad.any(), f"{what}: {bad.sum()} elements outside tolerance, max err {np.nanmax(err):.3e}"


def assert_bits(got, want, what):
    got = np.ascontiguousarray(got, np.float32)
    want = np.ascontiguousarray(want, np.float32)
    assert got.shape == want.shape, what
    diff = got.view(np.uint32) != want.view(np.uint32)
    assert not diff.any(), f"{what}: {diff.sum()} of {diff.size} elements differ in bits"

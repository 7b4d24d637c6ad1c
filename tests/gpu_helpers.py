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


SEQ_MAX = 32  # MLKV_SEQ_SEGMENT_MAX


class CountTracker:
    """Largest per-step occurrence count of every key seen in apply batches."""

    def __init__(self):
        self.max_count = {}

    def add(self, keys):
        u, c = np.unique(np.asarray(keys), return_counts=True)
        for k, n in zip(u.tolist(), c.tolist()):
            if n > self.max_count.get(k, 0):
                self.max_count[k] = n

    def long_mask(self, keys):
        return np.array([self.max_count.get(int(k), 0) > SEQ_MAX for k in keys], bool)


def assert_table_parity(w, G, keys, ref32, ref64, tracker, what=""):
    """Rows and state of `keys` against the oracle.

    Keys whose every gradient segment was short are summed by the kernel in
    occurrence order with the oracle's fp32 op sequence: bit-exact against the
    fp32 oracle.  Keys that ever had a long segment are summed in chunks: within
    TOL of the fp64 oracle (exact sums), the benchmark spec's tolerance."""
    keys = np.asarray(keys)
    long_ = tracker.long_mask(keys)
    short = ~long_
    if short.any():
        rw, rG = ref32.export(keys[short])
        assert_bits(w[short], rw, f"{what} rows of short-segment keys vs fp32 oracle")
        assert_bits(G[short], rG, f"{what} state of short-segment keys vs fp32 oracle")
    if long_.any():
        rw, rG = ref64.export(keys[long_])
        assert_close(w[long_], rw, f"{what} rows of long-segment keys vs fp64 oracle")
        assert_close(G[long_], rG, f"{what} state of long-segment keys vs fp64 oracle")
    return int(short.sum()), int(long_.sum())

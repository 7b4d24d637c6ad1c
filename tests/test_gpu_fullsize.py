"""Parity at the workloads' full sizes, in the launch configuration bench.py times.

Each store is opened at its full capacity with max_batch = its step batch,
every key is preloaded, and full-size steps (Get, then the gradient apply)
run on the GPU.  The oracle cannot hold 10^8 rows, but keys are independent
under the method (a key's row depends only on its own lookups and
gradients), so the oracle is fed, step by step and in occurrence order, only
the lookups of a sample of keys: the hottest keys, random touched keys and
untouched keys.  Their rows, states and Get outputs are compared element by
element; key-to-row resolution is checked for every key on the device, and
the dedup counts of a full batch against the oracle's.
"""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import CountTracker, assert_bits, assert_close, assert_table_parity, host, torch_cuda

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

STEPS = 4
N_HOT, N_RANDOM, N_COLD = 24, 400, 16


# The tiered store in the benchmark's configuration: the host tier is scaled to
# the machine's host memory (96M rows x 1 KiB), with a 4M-row HBM cache.
TIER_ROWS, TIER_CACHE = 96_000_000, 4_000_000


def _config(name):
    cfg = W.ALL[name]()
    if name == "tiered":
        cfg.n_keys = TIER_ROWS
        cfg.hbm_cache_rows = TIER_CACHE
    return cfg


def _store(cfg):
    import os

    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    slot = 2 * ((cfg.dim + 7) // 8 * 8) * 4
    free, _ = torch.cuda.mem_get_info()
    dev_rows = cfg.hbm_cache_rows or cfg.n_keys
    need = dev_rows * slot + cfg.n_keys * 68 + (8 << 30)
    if free < need:
        pytest.skip(f"needs {need / 2**30:.0f} GiB of device memory")
    if cfg.hbm_cache_rows:
        host_free = os.sysconf("SC_AVPHYS_PAGES") * os.sysconf("SC_PAGE_SIZE")
        if host_free < cfg.n_keys * slot + (24 << 30):
            pytest.skip("not enough host memory for the host tier")
    return EmbeddingStore(dim=cfg.dim, capacity=cfg.n_keys, max_batch=cfg.batch, lr=cfg.lr, eps=cfg.eps,
                          state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
                          hbm_cache_rows=cfg.hbm_cache_rows, device="cuda:0")


def _oracles(cfg):
    kw = dict(lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi,
              seed=cfg.seed)
    return oracle.Table(cfg.dim, precision=32, **kw), oracle.Table(cfg.dim, precision=64, **kw)


@pytest.mark.parametrize("name", ["dlrm", "kg", "gnn", "tiered"])
def test_full_size_parity(name):
    torch = torch_cuda()
    cfg = _config(name)
    store = _store(cfg)
    dev = torch.device("cuda:0")
    # preload every key in preload order; row ids must be 0..n-1 in that order
    for s in range(0, cfg.n_keys, cfg.batch):
        store.insert(torch.from_numpy(cfg.preload_keys(s, s + cfg.batch)).to(dev))
    assert store.sync() == 0
    assert store.size() == cfg.n_keys
    for s in range(0, cfg.n_keys, cfg.batch):
        k = torch.from_numpy(cfg.preload_keys(s, s + cfg.batch)).to(dev)
        rows = store.find(k)
        want = torch.arange(s, s + k.numel(), device=dev, dtype=torch.int64)
        assert torch.equal(rows, want), f"key -> row mismatch in preload chunk at {s}"

    batches = [cfg.batch_keys(step) for step in range(STEPS + 1)]
    # sample: hottest keys of step 0, random touched keys, untouched keys
    u0, c0 = np.unique(batches[0], return_counts=True)
    hot = u0[np.argsort(-c0)[:N_HOT]]
    rng = np.random.default_rng(7)
    touched = np.unique(np.concatenate(batches[:STEPS]))
    rand = rng.choice(touched, N_RANDOM, replace=False)
    allk = cfg.preload_keys(0, min(cfg.n_keys, 4_000_000))
    cold = rng.choice(np.setdiff1d(allk, touched)[:100_000], N_COLD, replace=False)
    sample = np.unique(np.concatenate([hot, rand, cold]))
    ref32, ref64 = _oracles(cfg)
    ref32.insert(sample)
    ref64.insert(sample)
    tracker = CountTracker()

    out = torch.empty((cfg.batch, cfg.dim), dtype=torch.float32, device=dev)
    for step, keys in enumerate(batches[:STEPS]):
        grads = cfg.grads(step)
        kd = torch.from_numpy(keys).to(dev)
        store.get(kd, out=out)
        sel = np.nonzero(np.isin(keys, sample))[0]  # occurrence order
        got = host(out[torch.from_numpy(sel).to(dev)])
        want, _, _ = ref32.get(keys[sel])
        want64, _, _ = ref64.get(keys[sel])
        exact = ~tracker.long_mask(keys[sel])
        assert_bits(got[exact], want[exact], f"{name} Get step {step} (short-run keys)")
        assert_close(got[~exact], want64[~exact], f"{name} Get step {step} (long-run keys)")
        if step == 0:
            # Get is a bit-exact copy of the stored rows, on the whole batch
            w_now, _ = store.export(kd)
            assert torch.equal(out.view(torch.int32), w_now.view(torch.int32))
        if cfg.hbm_cache_rows:  # the next batch is prefetched beside this apply
            nxt = torch.from_numpy(batches[step + 1]).to(dev)
            store.lookahead(nxt)
        store.apply_grad(kd, torch.from_numpy(grads).to(dev))
        ref32.apply_grad(keys[sel], grads[sel])
        ref64.apply_grad(keys[sel], grads[sel])
        tracker.add(keys[sel])
        del grads
    assert store.sync() == 0
    w, G = store.export(torch.from_numpy(sample).to(dev))
    n_short, n_long = assert_table_parity(host(w), host(G), sample, ref32, ref64, tracker, what=name)
    assert n_long >= 1 and n_short >= N_RANDOM // 2
    # untouched keys still hold their init rows, bit for bit
    cw, cG = store.export(torch.from_numpy(cold).to(dev))
    rw, rG = ref32.export(cold)
    assert_bits(host(cw), rw, f"{name} untouched rows")

    # dedup counts of a full batch, bit-exact against the oracle
    uniq, counts = store.dedup(torch.from_numpy(batches[0]).to(dev))
    uniq, counts = host(uniq), host(counts)
    ou, oc, _ = oracle.dedup(batches[0])
    o, g = np.argsort(ou), np.argsort(uniq)
    assert np.array_equal(uniq[g], ou[o]) and np.array_equal(counts[g].astype(np.int64), oc[o])
    assert store.last_unique() == len(ou)
    if cfg.hbm_cache_rows:
        fetched, _, _ = store.tier_stats()
        assert fetched > 0
    store.close()

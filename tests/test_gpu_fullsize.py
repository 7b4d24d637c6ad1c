"""Parity at the workloads' full sizes and full step counts, in the launch
configuration bench.py times.

Each store is opened at its full capacity with max_batch = its step batch,
every key is preloaded, and the workload's whole run (DLRM and KG 50 steps,
GNN 30, tiered 20) of full-size steps (Get, then the gradient apply) runs on
the GPU.  The oracle cannot hold 10^8 rows, but keys are independent under the
method (a key's row depends only on its own lookups and gradients), so the
oracle is fed, step by step and in occurrence order, only the lookups of a
sample of keys:

  * every key whose lookups in some step number more than MLKV_SEQ_SEGMENT_MAX
    (the long runs, summed in compensated chunks: the only keys whose sums are
    not the sequential fp32 ones) -- followed by the fp64 oracle;
  * random touched keys, keys with short runs of several lookups and
    untouched keys -- followed by the fp32 oracle.

At every step each sampled key's Get output is compared with the oracle's, and
after the last step its row and state:
  * keys whose runs were all short: bit for bit against the fp32 oracle (the
    kernel sums them in occurrence order with the same op sequence);
  * keys whose runs were all long: within 1e-5 * (1 + |ref|) of the fp64
    oracle;
  * keys with short runs in some steps and long runs in others (summed
    sequentially in fp32 at the first, with compensation at the second): within
    1e-5 * (1 + |ref64|) + |ref32 - ref64| of the fp64 oracle, i.e. at most the
    tolerance beyond the distance of the sequential fp32 statement itself from
    fp64 (that distance is large only where an Adagrad step is ill-conditioned,
    a summed gradient element near eps on a fresh state).
On the device every lookup's output equals the output of its key's first
lookup.  Key-to-row resolution is checked for every key on the device, and the
dedup counts of a full batch against the oracle's.

Gradients are drawn on the device from a seeded generator (host generation of
50 x 872 MB would dominate the test); the rows the oracle needs are copied to
the host, so both sides see the same numbers.
"""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import SEQ_MAX, assert_bits, assert_close, host, torch_cuda

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_RANDOM, N_SHORT_MULTI, N_COLD = 400, 200, 16

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
    need = dev_rows * slot + cfg.n_keys * 68 + (12 << 30)
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


def _sample(cfg, batches, steps):
    """(keys with only long runs, keys with long and short runs, a sample of
    keys with only short runs, untouched keys) of the run."""
    rng = np.random.default_rng(7)
    long_keys, short_keys, touched, multi = [], [], [], None
    for s in range(steps):
        u, c = np.unique(batches[s], return_counts=True)
        long_keys.append(u[c > SEQ_MAX])
        short_keys.append(u[c <= SEQ_MAX])
        touched.append(u)
        if s == 0:
            multi = u[(c >= 2) & (c <= SEQ_MAX)]
    long_keys = np.unique(np.concatenate(long_keys))
    mixed = np.intersect1d(long_keys, np.unique(np.concatenate(short_keys)), assume_unique=True)
    pure_long = np.setdiff1d(long_keys, mixed, assume_unique=True)
    touched = np.unique(np.concatenate(touched))
    short_pool = np.setdiff1d(touched, long_keys, assume_unique=True)
    rand = rng.choice(short_pool, min(N_RANDOM, len(short_pool)), replace=False)
    multi = np.setdiff1d(multi, long_keys, assume_unique=True)
    multi = rng.choice(multi, min(N_SHORT_MULTI, len(multi)), replace=False) if len(multi) else multi
    allk = cfg.preload_keys(0, min(cfg.n_keys, 4_000_000))
    cold = rng.choice(np.setdiff1d(allk, touched)[:100_000], N_COLD, replace=False)
    return pure_long, mixed, np.unique(np.concatenate([rand, multi])), cold


def _assert_mixed(got, want64, want32, what):
    """Within the fp64 tolerance widened by the fp32 oracle's own distance from fp64."""
    got, r64, r32 = (np.asarray(x, np.float64) for x in (got, want64, want32))
    err = np.abs(got - r64)
    bound = 1e-5 * (1.0 + np.abs(r64)) + np.abs(r32 - r64)
    bad = ~(err <= bound)
    assert not bad.any(), f"{what}: {bad.sum()} elements outside the bound, max err {np.nanmax(err):.3e}"


@pytest.mark.parametrize("name", ["dlrm", "kg", "gnn", "tiered"])
def test_full_size_parity(name):
    torch = torch_cuda()
    cfg = _config(name)
    steps = cfg.steps
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

    batches = [cfg.batch_keys(step) for step in range(steps + 1)]
    pure_long, mixed, short_keys, cold = _sample(cfg, batches, steps)
    assert len(pure_long) + len(mixed) >= 1 and len(short_keys) >= N_RANDOM // 2
    keys32 = np.concatenate([short_keys, mixed])  # lookups the fp32 oracle follows
    keys64 = np.concatenate([pure_long, mixed])   # ... and the fp64 oracle
    ref32, ref64 = _oracles(cfg)
    ref32.insert(np.concatenate([keys32, cold]))
    ref64.insert(keys64)
    # each oracle runs on its own host thread, in call order (ctypes releases the
    # GIL), beside the GPU steps
    ex32, ex64 = ThreadPoolExecutor(1), ThreadPoolExecutor(1)
    pending = []
    applies = []  # the oracles' apply futures: the loop stays a few steps ahead of them at most

    def check_gets(what, got, f32, f64, mode):
        r32 = f32.result() if f32 is not None else None
        r64 = f64.result() if f64 is not None else None
        for r in (r32, r64):
            assert r is None or r[2] == 0, what
        if mode == "short":
            assert_bits(got, r32[0], what)
        elif mode == "long":
            assert_close(got, r64[0], what)
        else:
            _assert_mixed(got, r64[0], r32[0], what)

    out = torch.empty((cfg.batch, cfg.dim), dtype=torch.float32, device=dev)
    for step in range(steps):
        keys = batches[step]
        kd = torch.from_numpy(keys).to(dev)
        gd = cfg.grads_device(step, dev)
        store.get(kd, out=out)
        # every lookup of a key returns the same row: the output of its first lookup
        u, first, inv = np.unique(keys, return_index=True, return_inverse=True)
        first_of_pos = torch.from_numpy(first[inv]).to(dev)
        assert torch.equal(out.view(torch.int32), out[first_of_pos].view(torch.int32)), f"{name} step {step}"
        if step == 0:
            # Get is a bit-exact copy of the stored rows, on the whole batch
            w_now, _ = store.export(kd)
            assert torch.equal(out.view(torch.int32), w_now.view(torch.int32))
            del w_now
        # each sampled key's Get output at this step against the oracle's
        for ks, mode in ((short_keys, "short"), (pure_long, "long"), (mixed, "mixed")):
            m = np.isin(u, ks, assume_unique=True)
            if m.any():
                got = host(out[torch.from_numpy(first[m]).to(dev)])
                f32 = ex32.submit(ref32.get, u[m]) if mode != "long" else None
                f64 = ex64.submit(ref64.get, u[m]) if mode != "short" else None
                pending.append((f"{name} Get step {step} ({mode}-run keys)", got, f32, f64, mode))
        if cfg.hbm_cache_rows:  # the next batch is prefetched beside this apply
            store.lookahead(torch.from_numpy(batches[step + 1]).to(dev))
        store.apply_grad(kd, gd)
        while len(applies) > 4:
            assert applies.pop(0).result() == 0
        for ks, ex, ref in ((keys32, ex32, ref32), (keys64, ex64, ref64)):
            sel = np.nonzero(np.isin(keys, ks))[0]  # occurrence order
            if len(sel):
                g = host(gd[torch.from_numpy(sel).to(dev)])
                applies.append(ex.submit(ref.apply_grad, keys[sel], g))
        del gd
        while pending and all(f is None or f.done() for f in pending[0][2:4]):
            check_gets(*pending.pop(0))
    assert store.sync() == 0
    for f in applies:
        assert f.result() == 0
    for p in pending:
        check_gets(*p)
    ex32.shutdown()
    ex64.shutdown()

    # rows and state after the last step
    w, G = store.export(torch.from_numpy(short_keys).to(dev))
    rw, rG = ref32.export(short_keys)
    assert_bits(host(w), rw, f"{name} rows of short-run keys vs fp32 oracle")
    assert_bits(host(G), rG, f"{name} state of short-run keys vs fp32 oracle")
    if len(pure_long):
        w, G = store.export(torch.from_numpy(pure_long).to(dev))
        rw, rG = ref64.export(pure_long)
        assert_close(host(w), rw, f"{name} rows of long-run keys vs fp64 oracle")
        assert_close(host(G), rG, f"{name} state of long-run keys vs fp64 oracle")
    if len(mixed):
        w, G = store.export(torch.from_numpy(mixed).to(dev))
        rw, rG = ref64.export(mixed)
        sw, sG = ref32.export(mixed)
        _assert_mixed(host(w), rw, sw, f"{name} rows of mixed-run keys")
        _assert_mixed(host(G), rG, sG, f"{name} state of mixed-run keys")
    # untouched keys still hold their init rows, bit for bit
    cw, cG = store.export(torch.from_numpy(cold).to(dev))
    rw, rG = ref32.export(cold)
    assert_bits(host(cw), rw, f"{name} untouched rows")
    assert_bits(host(cG), rG, f"{name} untouched state")

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

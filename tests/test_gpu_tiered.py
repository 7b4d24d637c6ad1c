"""The tiered store (HBM cache over host memory, look-ahead on a side stream).

Caching changes where a row lives, never what it holds: every key's lookups
are still summed in occurrence order, so a tiered store must give the same
Gets, rows and states bit for bit as an HBM-resident store on the same steps,
with rows evicted (and written back) all the time when the cache is small.
"""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import CountTracker, assert_bits, assert_table_parity, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu


def _export(store, keys):
    """export in calls of at most max_batch keys"""
    ws, Gs = [], []
    for s in range(0, len(keys), store.max_batch):
        w, G = store.export(dev(keys[s:s + store.max_batch]))
        ws.append(host(w))
        Gs.append(host(G))
    return np.concatenate(ws), np.concatenate(Gs)


def _insert(store, keys):
    for s in range(0, len(keys), store.max_batch):
        store.insert(dev(keys[s:s + store.max_batch]))


def _stores(cfg, cache_rows):
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    kw = dict(dim=cfg.dim, capacity=cfg.n_keys, max_batch=cfg.batch, lr=cfg.lr, eps=cfg.eps,
              state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
              device=torch.device("cuda", 0))
    return EmbeddingStore(hbm_cache_rows=cache_rows, **kw), EmbeddingStore(**kw)


@pytest.mark.parametrize("lookahead", [False, True])
def test_tiered_matches_resident(lookahead):
    torch = torch_cuda()
    cfg = W.scaled(W.dlrm(), 100, 64)  # 26 x 40,000 rows, 26,624 lookups per step
    cache = 2 * cfg.batch + 4096
    tiered, resident = _stores(cfg, cache)
    for s in range(0, cfg.n_keys, cfg.batch):
        k = dev(cfg.preload_keys(s, s + cfg.batch))
        tiered.insert(k)
        resident.insert(k)
    steps = 8
    # half Zipf-hot lookups, half uniform over the whole table: ~13k new rows a
    # step, so the 57k-line cache overflows by step 5 and dirty rows go back
    rng = np.random.default_rng(11)
    pre = cfg.preload_keys()
    batches = []
    for s in range(steps + 1):
        b = cfg.batch_keys(s)
        b[1::2] = rng.choice(pre, len(b[1::2]))
        batches.append(b)
    for step in range(steps):
        kd = dev(batches[step])
        g = dev(cfg.grads(step))
        a = tiered.get(kd)
        b = resident.get(kd)
        assert_bits(host(a), host(b), f"Get step {step}")
        if lookahead:
            tiered.lookahead(dev(batches[step + 1]))
        tiered.apply_grad(kd, g)
        resident.apply_grad(kd, g)
        torch.cuda.synchronize()
    assert tiered.sync() == 0 and resident.sync() == 0
    touched = np.unique(np.concatenate(batches[:steps]))
    wt, Gt = _export(tiered, touched)
    wr, Gr = _export(resident, touched)
    assert_bits(wt, wr, "rows")
    assert_bits(Gt, Gr, "state")
    fetched, written, _ = tiered.tier_stats()
    assert fetched > cache and written > 0  # the cache overflowed and dirty rows went back
    # untouched keys read from the host tier
    cold = cfg.preload_keys(0, cfg.n_keys)[::997]
    assert_bits(_export(tiered, cold)[0], _export(resident, cold)[0], "host-tier rows")
    for s in range(0, len(touched), cfg.batch):
        part = dev(touched[s:s + cfg.batch])
        assert np.array_equal(host(tiered.find(part)), host(resident.find(part)))


def test_tiered_vs_oracle():
    torch_cuda()
    cfg = W.tiny()
    tiered, _ = _stores(cfg, 2 * cfg.batch + 1024)
    ref32 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=32)
    ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
    tracker = CountTracker()
    for step in range(cfg.steps):
        keys = cfg.batch_keys(step)
        grads = cfg.grads(step)
        out = host(tiered.get(dev(keys)))  # inserts on miss: new rows start in the host tier
        want, _, _ = ref32.get(keys)
        ref64.get(keys)
        exact = ~tracker.long_mask(keys)
        assert_bits(out[exact], want[exact], f"Get step {step}")
        if step + 1 < cfg.steps:
            tiered.lookahead(dev(cfg.batch_keys(step + 1)))
        tiered.apply_grad(dev(keys), dev(grads))
        ref32.apply_grad(keys, grads)
        ref64.apply_grad(keys, grads)
        tracker.add(keys)
    assert tiered.sync() == 0
    touched = np.unique(np.concatenate([cfg.batch_keys(s) for s in range(cfg.steps)]))
    w, G = _export(tiered, touched)
    assert_table_parity(w, G, touched, ref32, ref64, tracker, what="tiered")
    assert tiered.size() == ref32.size()


def test_apply_beside_lookahead_needs_the_preceding_get_keys():
    torch_cuda()
    cfg = W.scaled(W.tiny(), 10, 4)
    tiered, _ = _stores(cfg, 4 * cfg.batch)
    pre = cfg.preload_keys()
    _insert(tiered, pre)
    a, b, c = pre[:500], pre[500:1000], pre[1000:1500]
    g = np.zeros((500, cfg.dim), np.float32)
    tiered.get(dev(a))
    tiered.lookahead(dev(b))
    tiered.apply_grad(dev(a), dev(g))  # fine: the keys of the Get
    assert tiered.sync() == 0
    tiered.get(dev(a))
    tiered.lookahead(dev(b))
    tiered.apply_grad(dev(c), dev(g))  # keys the Get did not resolve
    assert tiered.sync() == 1


def test_open_rejects_small_cache():
    torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore, MLKVError

    with pytest.raises(MLKVError) as e:
        EmbeddingStore(dim=8, capacity=10_000, max_batch=1_000, hbm_cache_rows=1_500)
    assert e.value.code == 1

"""Edge cases and device-detected errors of the CUDA path (no GPU fault involved:
every error is a status the kernels record and the host reads)."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu


def _small(dim=8):
    cfg = W.scaled(W.tiny(), 1000, 100)
    cfg.dim = dim
    return cfg


def test_empty_and_max_batch():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import MLKVError

    cfg = _small()
    store, ref = make_pair(cfg, capacity=4096, max_batch=1000)
    empty = torch.empty(0, dtype=torch.int64, device="cuda:0")
    assert store.get(empty).shape == (0, cfg.dim)
    store.apply_grad(empty, torch.empty((0, cfg.dim), device="cuda:0"))
    store.put(empty, torch.empty((0, cfg.dim), device="cuda:0"))
    u, c = store.dedup(empty)
    assert u.numel() == 0
    assert store.size() == 0
    keys = np.arange(1000, dtype=np.int64) * 3 + 1
    out = host(store.get(dev(keys)))
    want, _, _ = ref.get(keys)
    assert_bits(out, want, "Get at max_batch")
    with pytest.raises(MLKVError) as e:
        store.get(dev(np.arange(1001, dtype=np.int64)))
    assert e.value.code == 1
    assert store.sync() == 0


def test_single_lookup():
    cfg = _small()
    store, ref = make_pair(cfg, capacity=16, max_batch=1)
    k = np.array([123456789], np.int64)
    assert_bits(host(store.get(dev(k))), ref.get(k)[0], "single Get")
    g = np.full((1, cfg.dim), 0.5, np.float32)
    store.apply_grad(dev(k), dev(g))
    ref.apply_grad(k, g)
    assert_bits(host(store.export(dev(k))[0]), ref.export(k)[0], "single apply")


@pytest.mark.parametrize("shape", ["all_distinct", "one_key", "every_length", "no_singletons", "small_runs"])
def test_run_length_mixes(shape):
    """Batches made only of runs of one lookup, of one long run, of runs of
    every length 1..40 (singletons, small and short runs, the 4/5 and 32/33
    boundaries, long runs), of no singletons at all, and of runs of 2-4 lookups
    at every offset of the 32-position windows (those that start in the last
    lanes of a window take their later positions from the next): rows and
    state against the oracle, and the apply's count of distinct rows
    (last_unique) against the batch's."""
    cfg = _small(dim=16)
    store, ref = make_pair(cfg, capacity=8192, max_batch=4096)
    rng = np.random.default_rng(11)
    if shape == "all_distinct":
        keys = rng.permutation(4096).astype(np.int64) * 7 + 3
    elif shape == "one_key":
        keys = np.full(4096, 99, np.int64)
    elif shape == "every_length":
        keys = np.concatenate([np.full(m, 1000 + m, np.int64) for m in range(1, 41)])
    elif shape == "small_runs":
        lens = rng.integers(2, 5, 1300)
        keys = np.repeat(np.arange(len(lens), dtype=np.int64) * 3 + 7, lens)
    else:
        keys = np.repeat(np.arange(2000, dtype=np.int64) * 5 + 1, 2)
    keys = keys[rng.permutation(len(keys))]  # occurrences scattered over the batch
    grads = (rng.standard_normal((len(keys), cfg.dim)) * 0.01).astype(np.float32)
    store.get(dev(keys))
    ref.get(keys)
    store.apply_grad(dev(keys), dev(grads))
    ref.apply_grad(keys, grads)
    assert store.sync() == 0
    u, c = np.unique(keys, return_counts=True)
    assert store.last_unique() == len(u)
    w, G = store.export(dev(u))
    rw, rG = ref.export(u)
    short = c <= 32  # summed in occurrence order: the oracle's op sequence, bit for bit
    assert_bits(host(w)[short], rw[short], f"{shape}: rows of short-run keys")
    assert_bits(host(G)[short], rG[short], f"{shape}: state of short-run keys")
    if (~short).any():
        ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                             init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
        ref64.get(keys)
        ref64.apply_grad(keys, grads)
        lw, lG = ref64.export(u[~short])
        tol = lambda got, want: np.abs(got - want) <= 1e-5 * (1 + np.abs(want))
        assert tol(host(w)[~short], lw).all() and tol(host(G)[~short], lG).all()


def test_not_found_without_insert():
    cfg = _small()
    store, ref = make_pair(cfg, capacity=64, max_batch=64, insert_on_miss=False)
    store.insert(dev(np.array([1, 2], np.int64)))
    out = host(store.get(dev(np.array([1, 3, 2], np.int64))))
    assert np.all(np.isnan(out[1])) and not np.isnan(out[[0, 2]]).any()
    assert store.sync() == 7
    assert store.size() == 2
    store.clear_status()
    assert store.sync() == 0


def test_reserved_key_is_rejected():
    cfg = _small()
    store, _ = make_pair(cfg, capacity=64, max_batch=64)
    out = host(store.get(dev(np.array([5, -1, 6], np.int64))))
    assert np.all(np.isnan(out[1]))
    assert store.sync() == 1
    store.clear_status()
    assert store.size() == 2


def test_capacity_full():
    from paper_2504_01506_gb300 import MLKVError

    cfg = _small()
    store, _ = make_pair(cfg, capacity=100, max_batch=256)
    store.insert(dev(np.arange(150, dtype=np.int64)))
    assert store.sync() == 5
    assert store.size() == 100
    # the first 100 distinct keys (first occurrence order) got rows 0..99
    store.clear_status()
    rows = host(store.find(dev(np.arange(150, dtype=np.int64))))
    assert rows[:100].tolist() == list(range(100)) and np.all(rows[100:] == -1)
    # a later call sees the sticky status once set again
    store.insert(dev(np.arange(200, 210, dtype=np.int64)))
    assert store.sync() == 5
    with pytest.raises(MLKVError):
        store.get(dev(np.arange(3, dtype=np.int64)))


def test_probe_limit_reported():
    torch_cuda()
    from paper_2504_01506_gb300._lib import IDENTITY_HASH, PROBE_LIMIT

    cfg = _small()
    store, _ = make_pair(cfg, capacity=4096, max_batch=4096, flags=IDENTITY_HASH)
    nslots = 8192
    keys = np.arange(PROBE_LIMIT + 200, dtype=np.int64) * nslots  # every key hashes to slot 0
    store.insert(dev(keys))
    assert store.sync() == 6
    store.clear_status()
    # slots 0 .. PROBE_LIMIT-1 went to PROBE_LIMIT of the keys (which ones is
    # up to the race for them); the rest ran out of probes and were not stored
    assert store.size() == PROBE_LIMIT
    found = host(store.find(dev(keys)))
    assert (found >= 0).sum() == PROBE_LIMIT
    assert sorted(found[found >= 0].tolist()) == list(range(PROBE_LIMIT))


def test_misaligned_buffers_use_scalar_path():
    torch = torch_cuda()
    cfg = _small(dim=16)
    store, ref = make_pair(cfg, capacity=256, max_batch=128)
    keys = np.arange(100, dtype=np.int64) * 5
    buf = torch.empty(100 * 16 + 1, dtype=torch.float32, device="cuda:0")
    out = buf[1:].view(100, 16)  # 4-byte offset: not 16-byte aligned
    store.get(dev(keys), out=out)
    assert_bits(host(out), ref.get(keys)[0], "Get into a misaligned buffer")
    g = (np.random.default_rng(1).standard_normal((100, 16)) * 0.01).astype(np.float32)
    gbuf = torch.empty(100 * 16 + 1, dtype=torch.float32, device="cuda:0")
    gbuf[1:].copy_(torch.from_numpy(g.reshape(-1)))
    store.apply_grad(dev(keys), gbuf[1:].view(100, 16))
    ref.apply_grad(keys, g)
    assert_bits(host(store.export(dev(keys))[0]), ref.export(keys)[0], "apply from a misaligned buffer")


def test_open_rejects_bad_configs():
    torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore, MLKVError

    for kw, code in ((dict(dim=0), 1), (dict(dim=1025), 1), (dict(dim=257), 1), (dict(capacity=0), 1),
                     (dict(staleness_bound=-1), 1),
                     (dict(staleness_bound=1, hbm_cache_rows=100), 2),  # stale-synchronous: HBM-resident only
                     (dict(staleness_bound=2**63 - 1, hbm_cache_rows=100), 2),
                     (dict(hbm_cache_rows=10), 1), (dict(flags=64), 1)):
        args = dict(dim=8, capacity=100, max_batch=10)
        args.update(kw)
        with pytest.raises(MLKVError) as e:
            EmbeddingStore(**args)
        assert e.value.code == code, kw


def test_lookahead_is_a_no_op_in_hbm():
    cfg = _small()
    store, ref = make_pair(cfg, capacity=512, max_batch=256)
    keys = np.arange(200, dtype=np.int64)
    store.insert(dev(keys))
    ref.insert(keys)
    before = host(store.get(dev(keys)))
    store.lookahead(dev(keys[::-1].copy()))
    after = host(store.get(dev(keys)))
    assert_bits(after, before, "Get after Lookahead")
    assert_bits(after, ref.get(keys)[0], "Get vs oracle")


def test_host_buffer_calls():
    torch = torch_cuda()
    cfg = W.scaled(W.tiny(), 10, 2)
    store, ref = make_pair(cfg)
    keys = cfg.batch_keys(0)
    grads = cfg.grads(0)
    hk = torch.from_numpy(keys).pin_memory()
    hout = torch.empty((len(keys), cfg.dim), dtype=torch.float32).pin_memory()
    store.get_host(hk, hout)
    torch.cuda.synchronize()
    assert_bits(hout.numpy(), ref.get(keys)[0], "host Get")
    store.apply_grad_host(hk, torch.from_numpy(grads).pin_memory())
    ref.apply_grad(keys, grads)
    torch.cuda.synchronize()
    uk = np.unique(keys)
    from gpu_helpers import assert_close

    assert_close(host(store.export(dev(uk))[0]), ref.export(uk)[0], "rows after host apply")

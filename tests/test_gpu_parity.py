"""CUDA path against the oracle, element by element, on seeded inputs."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import (CountTracker, assert_bits, assert_close, assert_table_parity, dev, host,
                         make_pair, torch_cuda)

pytestmark = pytest.mark.gpu


def test_init_rows_bit_exact():
    cfg = W.scaled(W.tiny(), 10, 4)
    store, ref = make_pair(cfg)
    keys = cfg.preload_keys()
    store.insert(dev(keys))
    ref.insert(keys)
    w, G = store.export(dev(keys))
    rw, rG = ref.export(keys)
    assert_bits(host(w), rw, "init rows")
    assert_bits(host(G), rG, "init state")
    assert store.size() == len(keys) == ref.size()


def test_tiny_config_full_parity():
    """Config: 100,000 keys, dim 16, 10 steps of 4,096 Zipf(1.05) lookups, Get then apply."""
    torch_cuda()
    cfg = W.tiny()
    store, ref32 = make_pair(cfg, precision=32)
    ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    ref32.insert(pre)
    ref64.insert(pre)
    # key -> row resolution: dense ids in preload order, bit-exact
    assert np.array_equal(host(store.find(dev(pre))), np.arange(len(pre)))
    max_count = {}
    tracker = CountTracker()
    tracker.max_count = max_count
    for step in range(cfg.steps):
        keys = cfg.batch_keys(step)
        grads = cfg.grads(step)
        out = host(store.get(dev(keys)))
        want, _, _ = ref32.get(keys)
        want64, _, _ = ref64.get(keys)
        # every step's Get against the oracle: keys whose runs so far were all
        # short bit for bit (fp32), the others within tolerance of fp64
        exact = ~tracker.long_mask(keys)
        assert_bits(out[exact], want[exact], f"Get of step {step} (short-run keys)")
        assert_close(out[~exact], want64[~exact], f"Get of step {step} (long-run keys)")
        if step == 0:
            assert_bits(out, want, "Get of step 0")
        # Get is a bit-exact copy of the store's own rows
        w_now, _ = store.export(dev(keys))
        assert_bits(out, host(w_now), f"Get vs export, step {step}")
        store.apply_grad(dev(keys), dev(grads))
        ref32.apply_grad(keys, grads)
        ref64.apply_grad(keys, grads)
        u, c = np.unique(keys, return_counts=True)
        for k, n in zip(u.tolist(), c.tolist()):
            max_count[k] = max(max_count.get(k, 0), n)
    assert store.sync() == 0
    w, G = store.export(dev(pre))
    n_short, n_long = assert_table_parity(host(w), host(G), pre, ref32, ref64, tracker)
    assert n_short > 0.99 * len(pre)
    assert store.size() == len(pre)


@pytest.mark.parametrize("d", [1, 3, 4, 16, 64, 100, 128, 256, 260, 1024])
def test_dims(d):
    cfg = W.scaled(W.tiny(), 100, 8)
    cfg.dim = d
    store, ref = make_pair(cfg)
    rng = np.random.default_rng(d)
    for step in range(3):
        keys = rng.integers(0, 300, 600) * 7919 + 11
        keys[:40] = 5  # one long segment
        grads = (rng.standard_normal((600, d)) * 0.01).astype(np.float32)
        out = host(store.get(dev(keys)))
        want, _, _ = ref.get(keys)
        (assert_bits if step == 0 else assert_close)(out, want, f"Get d={d}")
        store.apply_grad(dev(keys), dev(grads))
        ref.apply_grad(keys, grads)
    allk = np.unique(keys)
    w, G = store.export(dev(allk))
    rw, rG = ref.export(allk)
    assert_close(host(w), rw, f"rows d={d}")
    assert_close(host(G), rG, f"state d={d}")
    assert store.sync() == 0


def test_dedup_counts_bit_exact():
    cfg = W.tiny()
    store, _ = make_pair(cfg, insert_on_miss=True)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    cases = [cfg.batch_keys(s) for s in range(3)]
    cases += [np.full(4096, pre[7]), pre[:4096].copy(), pre[:1].copy(), pre[:4095].copy()]
    for keys in cases:
        uniq, counts = store.dedup(dev(keys))
        uniq, counts = host(uniq), host(counts)
        ou, oc, _ = oracle.dedup(keys)
        o = np.argsort(ou)
        g = np.argsort(uniq)
        assert np.array_equal(uniq[g], ou[o])
        assert np.array_equal(counts[g].astype(np.int64), oc[o])
        # ordered by row id
        rows = host(store.find(dev(uniq)))
        assert np.all(np.diff(rows) > 0)


def test_get_after_put_and_last_wins():
    cfg = W.scaled(W.tiny(), 100, 8)
    store, ref = make_pair(cfg)
    rng = np.random.default_rng(3)
    keys = rng.integers(0, 50, 400) + 1000
    vals = rng.standard_normal((400, cfg.dim)).astype(np.float32)
    store.put(dev(keys), dev(vals))
    ref.put(keys, vals)
    uk = np.unique(keys)
    out = host(store.get(dev(uk)))
    want, rows, _ = ref.get(uk)
    assert_bits(out, want, "Get after Put")
    assert np.array_equal(host(store.find(dev(uk))), rows)
    w, G = store.export(dev(uk))
    assert_bits(host(G), ref.export(uk)[1], "state after Put")
    # a second Put over present keys keeps their state
    store.apply_grad(dev(keys), dev(vals * 0.01))
    ref.apply_grad(keys, vals * 0.01)
    store.put(dev(uk[:10]), dev(vals[:10]))
    ref.put(uk[:10], vals[:10])
    w, G = store.export(dev(uk))
    rw, rG = ref.export(uk)
    assert_bits(host(w)[:10], rw[:10], "rows after re-Put")
    assert_close(host(G), rG, "state after re-Put")
    assert store.sync() == 0


def test_row_alloc_golden_on_gpu():
    """The hand-worked row ids of tests/golden/row_alloc.txt through the CUDA path."""
    import os

    torch_cuda()
    cfg = W.scaled(W.tiny(), 1000, 100)
    cfg.dim = 2
    store, _ = make_pair(cfg, capacity=64, max_batch=64)
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "row_alloc.txt")
    with open(path) as f:
        lines = [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]
    for ln in lines:
        lhs, rhs = ln.split("->")
        op, *ks = lhs.split()
        keys = np.array([int(x) for x in ks], np.int64)
        want = [int(x) for x in rhs.split()]
        if op == "size":
            assert store.size() == want[0], ln
            continue
        if op == "insert":
            store.insert(dev(keys))
        elif op == "get":
            store.get(dev(keys))
        elif op == "put":
            store.put(dev(keys), dev(np.ones((len(keys), 2), np.float32)))
        elif op == "apply":
            store.apply_grad(dev(keys), dev(np.ones((len(keys), 2), np.float32)))
        assert host(store.find(dev(keys))).tolist() == want, ln
    assert store.sync() == 0


def test_insert_on_miss_rows_match_oracle():
    cfg = W.tiny()
    store, ref = make_pair(cfg)
    long_keys = set()
    for step in range(4):
        keys = cfg.batch_keys(step)
        out = host(store.get(dev(keys)))
        want, rows, _ = ref.get(keys)
        # rows only ever summed in occurrence order are bit-exact; keys that had a
        # segment longer than MLKV_SEQ_SEGMENT_MAX are within tolerance
        exact = np.array([int(k) not in long_keys for k in keys])
        assert_bits(out[exact], want[exact], f"Get with inserts, step {step}")
        assert_close(out, want, f"Get with inserts, step {step}")
        assert np.array_equal(host(store.find(dev(keys))), rows)
        grads = cfg.grads(step)
        store.apply_grad(dev(keys), dev(grads))
        ref.apply_grad(keys, grads)
        u, c = np.unique(keys, return_counts=True)
        long_keys |= set(u[c > 32].tolist())
    assert store.size() == ref.size()
    assert store.sync() == 0


def test_long_segments():
    cfg = W.scaled(W.tiny(), 100, 1)
    cfg.dim = 128
    store, ref32 = make_pair(cfg, capacity=8192, max_batch=150_000)
    ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
    rng = np.random.default_rng(9)
    keys = np.concatenate([np.full(100_000, 77), np.full(5_000, 78), rng.integers(100, 5000, 20_000)])
    rng.shuffle(keys)
    grads = (rng.standard_normal((len(keys), 128)) * 1e-3).astype(np.float32)
    tracker = CountTracker()
    for _ in range(2):
        store.apply_grad(dev(keys), dev(grads))
        ref32.apply_grad(keys, grads)
        ref64.apply_grad(keys, grads)
        tracker.add(keys)
    uk = np.unique(keys)
    w, G = store.export(dev(uk))
    n_short, n_long = assert_table_parity(host(w), host(G), uk, ref32, ref64, tracker)
    assert n_long == 2 and n_short > 4000
    assert store.sync() == 0


def test_deterministic_runs():
    cfg = W.scaled(W.dlrm(), 200, 64)
    outs = []
    for _ in range(2):
        store, _ = make_pair(cfg)
        store.insert(dev(cfg.preload_keys()))
        for step in range(3):
            keys = cfg.batch_keys(step)
            store.get(dev(keys))
            store.apply_grad(dev(keys), dev(cfg.grads(step)))
        w, G = store.export(dev(cfg.preload_keys()))
        outs.append((host(w), host(G)))
        store.close()
    assert_bits(outs[0][0], outs[1][0], "rows run to run")
    assert_bits(outs[0][1], outs[1][1], "state run to run")


def test_apply_after_get_of_other_keys():
    """The gradient apply takes each position's row from the Get before it when
    the key there is the same, and probes otherwise: applies on keys that match
    the Get's only in part, on a shorter batch, on new keys, after a Put, and
    on keys absent from a store without insert-on-miss, all match the oracle."""
    torch_cuda()
    cfg = W.scaled(W.tiny(), 20, 4)  # 5,000 keys, 1,024 lookups, dim 16
    store, ref32 = make_pair(cfg, capacity=cfg.n_keys + 1_000, max_batch=cfg.n_keys + 1_000)  # room for new keys
    ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    ref32.insert(pre)
    ref64.insert(pre)
    rng = np.random.default_rng(3)
    tracker = CountTracker()
    touched = set(pre.tolist())

    def apply(keys, grads):
        store.apply_grad(dev(keys), dev(grads))
        ref32.apply_grad(keys, grads)
        ref64.apply_grad(keys, grads)
        tracker.add(keys)
        touched.update(np.asarray(keys).tolist())

    def get(keys):
        out = host(store.get(dev(keys)))
        want, _, _ = ref32.get(keys)
        ref64.get(keys)
        touched.update(np.asarray(keys).tolist())
        exact = ~tracker.long_mask(keys)
        assert_bits(out[exact], want[exact], "Get")

    for step in range(6):
        keys = cfg.batch_keys(step)
        grads = cfg.grads(step)
        get(keys)
        other = keys.copy()
        swap = rng.random(len(keys)) < 0.5
        other[swap] = rng.choice(pre, int(swap.sum()))          # present keys at other positions
        new = rng.random(len(keys)) < 0.05
        other[new] = (1 << 41) + step * 10_000 + np.arange(int(new.sum()))  # new keys
        if step % 2:
            other = other[: len(other) // 2]                     # a shorter batch
        apply(other, grads[: len(other)])
        if step == 3:  # a Put between a Get and the apply of its keys
            vals = (rng.standard_normal((len(keys), cfg.dim)) * 0.01).astype(np.float32)
            get(keys)
            store.put(dev(keys), dev(vals))
            ref32.put(keys, vals)
            ref64.put(keys, vals)
            apply(keys, grads)
    assert store.sync() == 0
    keys = np.array(sorted(touched), dtype=np.int64)
    w, G = store.export(dev(keys))
    assert_table_parity(host(w), host(G), keys, ref32, ref64, tracker, what="memo")
    assert store.size() == ref32.size()

    # without insert-on-miss: an absent key at a position the Get resolved is
    # skipped and reported, never given the Get's row
    store2, ref2 = make_pair(cfg, insert_on_miss=False)
    ref2_64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                           init_hi=cfg.init_hi, seed=cfg.seed, precision=64, insert_on_miss=False)
    store2.insert(dev(pre))
    ref2.insert(pre)
    ref2_64.insert(pre)
    keys = cfg.batch_keys(0)
    store2.get(dev(keys))
    absent = keys.copy()
    absent[::7] = (1 << 42) + np.arange(len(absent[::7]))
    store2.apply_grad(dev(absent), dev(cfg.grads(0)))
    ref2.apply_grad(absent, cfg.grads(0))
    ref2_64.apply_grad(absent, cfg.grads(0))
    assert store2.sync() == 7  # MLKV_ERR_NOT_FOUND
    store2.clear_status()
    w2, G2 = store2.export(dev(pre))
    tracker2 = CountTracker()
    tracker2.add(absent)
    assert_table_parity(host(w2), host(G2), pre, ref2, ref2_64, tracker2, what="without insert-on-miss")

"""Random sequences of every kind of call on one stream, with no synchronisation
between them, against the oracle.

Every kernel of the library may start while the kernel before it drains
(programmatic dependent launch) and waits for it on entry; calls also share the
table's scratch.  A missing wait or a scratch buffer reused too early shows up
here as a wrong Get, find, export or dedup output, or a wrong row at the end:
each output is kept on the device and checked only after the whole sequence
has been issued."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import CountTracker, assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu

TOL = 1e-5


def _close(got, want):
    return np.abs(np.asarray(got, np.float64) - want) <= TOL * (1 + np.abs(want))


@pytest.mark.parametrize("seed,dim,tiered", [(1, 32, False), (2, 16, False), (3, 100, False), (4, 32, True)])
def test_random_call_sequences(seed, dim, tiered):
    """The tiered case keeps its rows in host memory behind an HBM cache of
    two batches and a little more (batches of up to 1,024 lookups, 2,312 lines
    for 6,000 keys), so rows are evicted and fetched back all along; before some applies of the last Get's keys it issues a look-ahead of
    another batch (the training order Get, Lookahead, apply)."""
    torch = torch_cuda()
    cfg = W.scaled(W.tiny(), 10, 1)
    cfg.dim = dim
    n_keys, max_batch = 6_000, (1_024 if tiered else 4_096)
    store, ref32 = make_pair(cfg, capacity=20_000, max_batch=max_batch)
    if tiered:
        from paper_2504_01506_gb300 import EmbeddingStore

        store.close()
        store = EmbeddingStore(dim=cfg.dim, capacity=20_000, max_batch=max_batch, lr=cfg.lr, eps=cfg.eps,
                               state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
                               hbm_cache_rows=2 * max_batch + 64 + 200, device="cuda:0")  # < the 6,000 keys
    ref64 = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                         init_hi=cfg.init_hi, seed=cfg.seed, precision=64)
    rng = np.random.default_rng(seed)
    universe = rng.choice(1 << 40, n_keys, replace=False).astype(np.int64)
    weights = 1.0 / np.arange(1, n_keys + 1) ** 1.1
    weights /= weights.sum()
    tracker = CountTracker()
    checks = []  # (kind, device outputs, expected values, exact mask)
    last_get = None

    def batch():
        n = int(rng.integers(1, max_batch + 1))
        return universe[rng.choice(n_keys, n, p=weights)]

    prev = None
    la_pending = False  # a look-ahead was issued and no call has waited for it yet
    n_lookahead = 0
    for step in range(60):
        if step:
            prev = op
        op = rng.choice(["get", "apply", "apply_last", "put", "insert", "import", "find", "export", "dedup"],
                        p=[0.2, 0.15, 0.15, 0.1, 0.05, 0.05, 0.1, 0.1, 0.1])
        if op == "apply_last" and last_get is None:
            op = "get"
        if la_pending and op in ("apply", "apply_last"):
            op = "get"  # an apply would run beside the pending look-ahead too; every other call waits for it
        la_pending = la_pending and op in ("apply", "apply_last")
        if op == "get":
            keys = batch()
            out = store.get(dev(keys))
            want32, _, _ = ref32.get(keys)
            want64, _, _ = ref64.get(keys)
            checks.append(("get", (out,), (want32, want64), ~tracker.long_mask(keys)))
            last_get = keys
        elif op in ("apply", "apply_last"):
            keys = last_get if op == "apply_last" else batch()  # the training order, or other keys
            if tiered and op == "apply_last" and prev == "get" and rng.random() < 0.7:
                store.lookahead(dev(batch()))  # runs beside the apply, right after its Get
                la_pending = True
                n_lookahead += 1
            grads = (rng.standard_normal((len(keys), dim)) * 0.01).astype(np.float32)
            store.apply_grad(dev(keys), dev(grads))
            ref32.apply_grad(keys, grads)
            ref64.apply_grad(keys, grads)
            tracker.add(keys)
        elif op == "put":
            keys = batch()
            vals = (rng.standard_normal((len(keys), dim)) * 0.01).astype(np.float32)
            store.put(dev(keys), dev(vals))
            ref32.put(keys, vals)
            ref64.put(keys, vals)
        elif op == "insert":
            keys = universe[rng.choice(n_keys, int(rng.integers(1, max_batch // 2)))]
            store.insert(dev(keys))
            ref32.insert(keys)
            ref64.insert(keys)
        elif op == "import":
            keys = universe[rng.choice(n_keys, int(rng.integers(1, max_batch // 2)))]
            rows = (rng.standard_normal((len(keys), dim)) * 0.01).astype(np.float32)
            state = np.abs(rng.standard_normal((len(keys), dim)) * 0.01).astype(np.float32)
            store.import_(dev(keys), dev(rows), dev(state))
            ref32.import_(keys, rows, state)
            ref64.import_(keys, rows, state)
        elif op == "find":
            keys = batch()
            checks.append(("find", (store.find(dev(keys)),), (ref32.find(keys),), None))
        elif op == "export":
            keys = batch()
            w, G = store.export(dev(keys))
            rw32, rG32 = ref32.export(keys)
            rw64, rG64 = ref64.export(keys)
            checks.append(("export", (w, G), (rw32, rG32, rw64, rG64), ~tracker.long_mask(keys)))
        else:  # dedup without the host read of its count: raw call, checked at the end
            keys = batch()
            kd = dev(keys)
            n = len(keys)
            uniq = torch.empty(n, dtype=torch.int64, device="cuda:0")
            counts = torch.empty(n, dtype=torch.int32, device="cuda:0")
            num = torch.zeros(1, dtype=torch.int64, device="cuda:0")
            rc = store.lib.mlkv_dedup(store.h, kd.data_ptr(), n, uniq.data_ptr(), counts.data_ptr(),
                                      num.data_ptr(), torch.cuda.current_stream().cuda_stream)
            assert rc == 0
            present = ref32.find(keys) >= 0
            ou, oc, _ = oracle.dedup(keys[present])
            checks.append(("dedup", (uniq, counts, num, kd), (ou, oc), None))

    assert store.sync() == 0
    if tiered:  # the case did what it is for: look-aheads, and rows evicted and fetched back
        fetched, written, _ = store.tier_stats()
        assert n_lookahead >= 2 and fetched > 0 and written > 0, (n_lookahead, fetched, written)
    for i, (kind, got, want, exact) in enumerate(checks):
        what = f"seed {seed}, dim {dim}, check {i} ({kind})"
        if kind == "get":
            out = host(got[0])
            assert_bits(out[exact], want[0][exact], what)
            assert _close(out[~exact], want[1][~exact]).all(), what
        elif kind == "find":
            assert np.array_equal(host(got[0]), want[0]), what
        elif kind == "export":
            w, G = host(got[0]), host(got[1])
            assert_bits(w[exact], want[0][exact], what + " rows")
            assert_bits(G[exact], want[1][exact], what + " state")
            assert _close(w[~exact], want[2][~exact]).all() and _close(G[~exact], want[3][~exact]).all(), what
        else:
            u = int(host(got[2])[0])
            uniq, counts = host(got[0])[:u], host(got[1])[:u]
            ou, oc = want
            o, g = np.argsort(ou), np.argsort(uniq)
            assert u == len(ou), what
            assert np.array_equal(uniq[g], ou[o]) and np.array_equal(counts[g].astype(np.int64), oc[o]), what
    # the whole table at the end
    keys = ref32.keys()
    assert store.size() == len(keys)
    assert np.array_equal(host(store.keys()), keys)
    parts = [store.export(dev(keys[i:i + max_batch])) for i in range(0, len(keys), max_batch)]
    w = torch.cat([p[0] for p in parts])
    G = torch.cat([p[1] for p in parts])
    exact = ~tracker.long_mask(keys)
    rw32, rG32 = ref32.export(keys)
    rw64, rG64 = ref64.export(keys)
    assert_bits(host(w)[exact], rw32[exact], "final rows")
    assert_bits(host(G)[exact], rG32[exact], "final state")
    assert _close(host(w)[~exact], rw64[~exact]).all() and _close(host(G)[~exact], rG64[~exact]).all()

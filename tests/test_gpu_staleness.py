"""Stale-synchronous and asynchronous tables (the bounded staleness of MLKV
Section 3.3.1): Gets on one stream, gradient applies on another, against the
oracle.

With bound s a Get may run beside the last s applies issued before it: each
element it returns is the oracle's value after j applies, for some j between
(t - s) and t at step t, chosen element by element (any j <= t with no bound,
the asynchronous mode).  The applies themselves run
in order, so the table after the last one is exactly the bulk-synchronous
oracle's.  Batches draw keys uniformly (no run longer than 32 lookups), so every
comparison is bit for bit against the fp32 oracle."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import assert_bits, dev, host, torch_cuda

pytestmark = pytest.mark.gpu

DIM, N_KEYS, BATCH, STEPS = 16, 5_000, 1_024, 10
ASYNC = 2**63 - 1


def _store(cfg, s, **over):
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    kw = dict(dim=DIM, capacity=N_KEYS + 2_000, max_batch=8_192, lr=cfg.lr, eps=cfg.eps,
              state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
              staleness_bound=s, device=torch.device("cuda", 0))
    kw.update(over)
    return EmbeddingStore(**kw)


def _oracle(cfg):
    return oracle.Table(DIM, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                        init_hi=cfg.init_hi, seed=cfg.seed, precision=32)


@pytest.mark.parametrize("s,host_buffers", [(1, False), (2, False), (1, True), (100, False), (ASYNC, False)])
def test_stale_synchronous_training_loop(s, host_buffers):
    """host_buffers: the host-buffer calls, whose keys and gradients are staged
    on the device inside the call (a Get's staging must not be an apply's)."""
    torch = torch_cuda()
    cfg = W.tiny()
    rng = np.random.default_rng(40 + s)
    pre = rng.choice(1 << 40, N_KEYS, replace=False).astype(np.int64)
    steps = []
    for t in range(STEPS):
        keys = pre[rng.integers(0, N_KEYS, BATCH)]
        new = rng.random(BATCH) < 0.05  # new keys: inserted by the Get, beside an apply
        keys[new] = (1 << 41) + t * 1_000 + np.arange(int(new.sum()))
        grads = (rng.standard_normal((BATCH, DIM)) * 0.01).astype(np.float32)
        steps.append((keys, grads))

    # the bulk-synchronous oracle, with every key's value after each apply count
    ref = _oracle(cfg)
    ref.insert(pre)
    snaps = []  # snaps[j]: {key: row} after j applies (and the j-th Get's inserts)
    for keys, grads in steps:
        ref.get(keys)
        allk = ref.keys()
        w, _ = ref.export(allk)
        snaps.append(dict(zip(allk.tolist(), w)))
        ref.apply_grad(keys, grads)
    allk = ref.keys()
    final_w, final_G = ref.export(allk)

    store = _store(cfg, s)
    store.insert(dev(pre))
    if host_buffers:
        kd = [torch.from_numpy(k).pin_memory() for k, _ in steps]
        gd = [torch.from_numpy(g).pin_memory() for _, g in steps]
        outs = [torch.empty((BATCH, DIM)).pin_memory() for _ in steps]
    else:
        kd = [dev(k) for k, _ in steps]
        gd = [dev(g) for _, g in steps]
        outs = [torch.empty((BATCH, DIM), device="cuda:0") for _ in steps]
    torch.cuda.synchronize()
    s_get, s_apply = torch.cuda.Stream(), torch.cuda.Stream()
    for t in range(STEPS):
        with torch.cuda.stream(s_get):
            if host_buffers:
                store.get_host(kd[t], outs[t])
            else:
                store.get(kd[t], out=outs[t])
        with torch.cuda.stream(s_apply):
            if host_buffers:
                store.apply_grad_host(kd[t], gd[t])
            else:
                store.apply_grad(kd[t], gd[t])
    torch.cuda.synchronize()
    assert store.sync() == 0

    # after the last apply: exactly the bulk-synchronous table
    w, G = store.export(dev(allk))
    assert_bits(host(w), final_w, f"s={s}: rows after the last apply")
    assert_bits(host(G), final_G, f"s={s}: state after the last apply")
    assert store.size() == len(allk)

    # every element of Get(t) is the value after j applies, t - s <= j <= t
    first = {}  # a key's row when first inserted (its value at every earlier apply count)
    for snap in snaps:
        for k, row in snap.items():
            first.setdefault(k, row)
    for t, (keys, _) in enumerate(steps):
        got = outs[t].numpy() if host_buffers else host(outs[t])
        ok = np.zeros_like(got, dtype=bool)
        for j in range(max(0, t - s), t + 1):  # (s above 64 is kept as 64: within the bound too)
            want = np.stack([snaps[j].get(k, first[k]) for k in keys.tolist()])
            ok |= got.view(np.int32) == want.view(np.int32)
        assert ok.all(), f"s={s}, step {t}: {int((~ok).sum())} elements outside the staleness bound"


def test_stale_synchronous_apply_inserts_nothing():
    """An apply of a stale-synchronous table skips absent keys (a Get beside it
    may be inserting) and reports them."""
    cfg = W.tiny()
    store = _store(cfg, 1)
    ref = _oracle(cfg)
    keys = np.arange(100, dtype=np.int64) * 7 + 1
    store.insert(dev(keys))
    ref.insert(keys)
    absent = keys.copy()
    absent[::10] = (1 << 42) + np.arange(10)
    grads = np.full((100, DIM), 0.01, np.float32)
    store.apply_grad(dev(absent), dev(grads))
    assert store.sync() == 7  # MLKV_ERR_NOT_FOUND
    store.clear_status()
    assert store.size() == 100
    present = np.isin(absent, keys)
    ref.apply_grad(absent[present], grads[present])
    w, _ = store.export(dev(keys))
    assert_bits(host(w), ref.export(keys)[0], "rows of the present keys")


@pytest.mark.filterwarnings("ignore:The CUDA Graph is empty")  # the refused capture records nothing
def test_stale_synchronous_calls_refuse_capture():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import MLKVError

    store = _store(W.tiny(), 1)
    keys = dev(np.arange(10, dtype=np.int64) + 1)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with pytest.raises(MLKVError) as e:
        with torch.cuda.stream(s):
            with torch.cuda.graph(graph, stream=s):
                store.get(keys)
    assert e.value.code == 2  # MLKV_ERR_UNSUPPORTED

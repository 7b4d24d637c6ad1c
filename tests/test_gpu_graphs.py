"""Captured CUDA graphs of store calls against the same calls made one by one.

Every call's work is device-driven (miss counts, runs, long runs are found on
the GPU), so a captured sequence replayed with the same pointers must give the
same Gets, rows and states bit for bit as the plain calls, for any number of
calls per graph."""
import numpy as np
import pytest

import workloads as W
from gpu_helpers import assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu


def test_graph_replay_matches_plain_calls():
    torch = torch_cuda()
    cfg = W.scaled(W.tiny(), 10, 4)  # 10,000 keys, 1,024 lookups, dim 16
    plain, _ = make_pair(cfg, capacity=cfg.n_keys + 4_000, max_batch=cfg.n_keys + 4_000)
    graphed, _ = make_pair(cfg, capacity=cfg.n_keys + 4_000, max_batch=cfg.n_keys + 4_000)
    pre = cfg.preload_keys()
    plain.insert(dev(pre))
    graphed.insert(dev(pre))
    k0, k1 = cfg.batch_keys(0), cfg.batch_keys(1)
    k1[::50] = (1 << 40) + np.arange(len(k1[::50]))  # new keys: the miss path runs inside the graph
    g0 = dev(cfg.grads(0))
    kd0, kd1 = dev(k0), dev(k1)
    outs = {name: (torch.empty((len(k0), cfg.dim), device="cuda"), torch.empty((len(k1), cfg.dim), device="cuda"))
            for name in ("plain", "graphed")}

    def calls(store, o):  # three calls: an odd number per graph
        store.get(kd0, out=o[0])
        store.apply_grad(kd0, g0)
        store.get(kd1, out=o[1])

    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            calls(graphed, outs["graphed"])
    torch.cuda.synchronize()
    for rep in range(4):
        graph.replay()
        calls(plain, outs["plain"])
        torch.cuda.synchronize()
        assert_bits(host(outs["graphed"][0]), host(outs["plain"][0]), f"Get 0, replay {rep}")
        assert_bits(host(outs["graphed"][1]), host(outs["plain"][1]), f"Get 1, replay {rep}")
    assert graphed.sync() == 0 and plain.sync() == 0
    keys = np.unique(np.concatenate([pre, k1]))
    wg, Gg = graphed.export(dev(keys))
    wp, Gp = plain.export(dev(keys))
    assert_bits(host(wg), host(wp), "rows")
    assert_bits(host(Gg), host(Gp), "state")
    assert graphed.size() == plain.size()


@pytest.mark.filterwarnings("ignore:The CUDA Graph is empty")  # the refused capture records nothing
def test_tiered_calls_refuse_capture():
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore, MLKVError

    cfg = W.scaled(W.tiny(), 10, 4)
    store = EmbeddingStore(dim=cfg.dim, capacity=cfg.n_keys, max_batch=cfg.batch,
                           hbm_cache_rows=2 * cfg.batch + 4096, device=torch.device("cuda", 0))
    keys = dev(cfg.batch_keys(0))
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with pytest.raises(MLKVError) as e:
        with torch.cuda.stream(s):
            with torch.cuda.graph(graph, stream=s):
                store.get(keys)
    assert e.value.code == 2  # MLKV_ERR_UNSUPPORTED
    store.clear_status()
    store.get(keys)  # still usable after the refused capture
    assert store.sync() == 0


@pytest.mark.parametrize("last", [0, 1])
def test_direct_calls_after_replays(last):
    """Replays do not pass through the host, so the host cannot tell which
    counters the last replayed call left set.  Two graphs are captured (one
    per counter copy), replayed in either order, and then the same kind of
    calls is made directly: the table must match one driven by direct calls
    only, and the oracle.  The batch is mostly runs of one lookup and
    max_batch is its size, so a run list counted twice would run past its end."""
    torch = torch_cuda()
    import oracle

    rng = np.random.default_rng(31 + last)
    n = 3000
    cfg = W.scaled(W.tiny(), 20, 1)
    cfg.batch = n
    graphed, ref = make_pair(cfg, capacity=cfg.n_keys, max_batch=n)
    plain, _ = make_pair(cfg, capacity=cfg.n_keys, max_batch=n)
    pre = cfg.preload_keys()
    for st in (graphed, plain):
        st.insert(dev(pre[:n]))
        st.insert(dev(pre[n:]))
    ref.insert(pre)
    batches = []
    for b in range(4):
        k = rng.choice(pre, n, replace=False)
        k[:300] = k[300:600]  # a few runs of two; the rest runs of one
        batches.append((k, (rng.standard_normal((n, cfg.dim)) * 0.01).astype(np.float32)))
    kd = [dev(k) for k, _ in batches]
    gd = [dev(g) for _, g in batches]
    outs = [torch.empty((n, cfg.dim), device="cuda") for _ in batches]
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    graphs = []
    with torch.cuda.stream(s):
        for j in range(2):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                graphed.get(kd[j], out=outs[j])
                graphed.apply_grad(kd[j], gd[j])
            graphs.append(g)
    torch.cuda.synchronize()
    order = [1 - last, last]
    for j in order:  # replays, the last one `last`
        graphs[j].replay()
    for j in (2, 3):  # then direct calls
        graphed.get(kd[j], out=outs[j])
        graphed.apply_grad(kd[j], gd[j])
    assert graphed.sync() == 0
    for j in order + [2, 3]:  # the same calls, made directly, and in the oracle
        want = plain.get(kd[j])
        plain.apply_grad(kd[j], gd[j])
        k, g = batches[j]
        rw, _, _ = ref.get(k)
        ref.apply_grad(k, g)
        if j >= 2:
            assert_bits(host(outs[j]), host(want), f"Get of direct call {j}")
            assert_bits(host(outs[j]), rw, f"Get of direct call {j} vs oracle")
    assert plain.sync() == 0

    def export(store):  # max_batch keys at a time
        parts = [store.export(dev(pre[i:i + n])) for i in range(0, len(pre), n)]
        return (np.concatenate([host(p[0]) for p in parts]), np.concatenate([host(p[1]) for p in parts]))

    (w, G), (pw, pG) = export(graphed), export(plain)
    rw, rG = ref.export(pre)
    assert_bits(w, pw, "rows vs direct calls only")
    assert_bits(G, pG, "state vs direct calls only")
    assert_bits(w, rw, "rows vs oracle")
    assert_bits(G, rG, "state vs oracle")

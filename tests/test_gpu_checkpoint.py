"""Checkpoints: the table's keys in row order, import of rows and state, and a
restore that continues bit-identically (MLKV Section 2.2 keeps data by
periodic checkpoints; the oracle's oracle_keys / oracle_import state what a
checkpoint holds and what a restore does)."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu


def _cfg():
    return W.scaled(W.tiny(), 20, 4)  # 5,000 keys, 1,024 lookups, dim 16


def test_keys_and_import_match_the_oracle():
    torch_cuda()
    cfg = _cfg()
    store, ref = make_pair(cfg, capacity=cfg.n_keys + 2_000, max_batch=cfg.n_keys + 2_000)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    ref.insert(pre)
    for step in range(3):
        keys = cfg.batch_keys(step)
        keys[::40] = (1 << 41) + step * 1_000 + np.arange(len(keys[::40]))  # new keys: rows by first occurrence
        store.get(dev(keys))
        ref.get(keys)
        store.apply_grad(dev(keys), dev(cfg.grads(step)))
        ref.apply_grad(keys, cfg.grads(step))
    assert store.sync() == 0
    assert np.array_equal(host(store.keys()), ref.keys())
    rng = np.random.default_rng(4)
    ik = np.concatenate([pre[:300], (1 << 42) + np.arange(50), pre[:10]])  # present, new, duplicates
    rows = rng.standard_normal((len(ik), cfg.dim)).astype(np.float32)
    state = np.abs(rng.standard_normal((len(ik), cfg.dim))).astype(np.float32)
    store.import_(dev(ik), dev(rows), dev(state))
    ref.import_(ik, rows, state)
    nk = (1 << 43) + np.arange(20)
    store.import_(dev(nk), dev(rows[:20]))  # no state: state_init for new keys
    ref.import_(nk, rows[:20])
    assert store.sync() == 0
    allk = ref.keys()
    assert np.array_equal(host(store.keys()), allk)
    w, G = store.export(dev(allk))
    rw, rG = ref.export(allk)
    imported = np.isin(allk, np.concatenate([ik, nk]))
    assert_bits(host(w)[imported], rw[imported], "imported rows")
    assert_bits(host(G)[imported], rG[imported], "imported state")


def test_restore_continues_bit_identically(tmp_path):
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    cfg = _cfg()
    kw = dict(dim=cfg.dim, capacity=cfg.n_keys + 2_000, max_batch=cfg.n_keys + 2_000, lr=cfg.lr, eps=cfg.eps,
              state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
              device=torch.device("cuda", 0))
    a = EmbeddingStore(**kw)
    a.insert(dev(cfg.preload_keys()))
    batches = []
    for step in range(10):
        keys = cfg.batch_keys(step)
        keys[::50] = (1 << 41) + step * 1_000 + np.arange(len(keys[::50]))
        batches.append((keys, cfg.grads(step)))
    for keys, g in batches[:5]:
        a.get(dev(keys))
        a.apply_grad(dev(keys), dev(g))
    path = str(tmp_path / "ckpt.npz")
    a.save(path)
    b = EmbeddingStore(**kw)
    b.load(path)
    assert b.size() == a.size()
    assert np.array_equal(host(b.keys()), host(a.keys()))
    assert np.array_equal(host(b.find(a.keys())), np.arange(a.size()))  # the same row ids
    for step, (keys, g) in enumerate(batches[5:], start=5):
        assert_bits(host(b.get(dev(keys))), host(a.get(dev(keys))), f"Get step {step}")
        a.apply_grad(dev(keys), dev(g))
        b.apply_grad(dev(keys), dev(g))
    assert a.sync() == 0 and b.sync() == 0
    keys = a.keys()
    wa, Ga = a.export(keys)
    wb, Gb = b.export(keys)
    assert_bits(host(wb), host(wa), "rows after the restored run")
    assert_bits(host(Gb), host(Ga), "state after the restored run")


def test_tiered_checkpoint_loads_into_an_hbm_table(tmp_path):
    torch = torch_cuda()
    from paper_2504_01506_gb300 import EmbeddingStore

    cfg = _cfg()
    kw = dict(dim=cfg.dim, capacity=cfg.n_keys, max_batch=cfg.n_keys, lr=cfg.lr, eps=cfg.eps,
              state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
              device=torch.device("cuda", 0))
    tiered = EmbeddingStore(hbm_cache_rows=2 * cfg.n_keys + 64, **kw)
    tiered.insert(dev(cfg.preload_keys()))
    for step in range(4):
        keys = dev(cfg.batch_keys(step))
        tiered.get(keys)
        tiered.apply_grad(keys, dev(cfg.grads(step)))
    path = str(tmp_path / "tiered.npz")
    tiered.save(path)
    hbm = EmbeddingStore(**kw)
    hbm.load(path)
    keys = tiered.keys()
    assert np.array_equal(host(hbm.keys()), host(keys))
    wt, Gt = tiered.export(keys)
    wh, Gh = hbm.export(keys)
    assert_bits(host(wh), host(wt), "rows")
    assert_bits(host(Gh), host(Gt), "state")

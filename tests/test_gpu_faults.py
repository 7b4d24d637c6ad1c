"""Error paths under host-side fault injection (mlkv_debug_fail).

A failed allocation or copy is made on the host: the library's own allocation
and copy helpers return an error without calling CUDA, so nothing faults on the
GPU.  Checked: every allocation mlkv_open makes, failed in turn, gives
MLKV_ERR_NOMEM, a null handle and no device memory left behind (HBM-resident
and tiered tables); a failed staging allocation or copy of a host-buffer call
returns its error, applies nothing and leaves the table usable; a bounded
wait inside a kernel (the grid barriers of the kernel that gives new keys their
rows) made to run out returns MLKV_ERR_TIMEOUT within seconds, the context
stays usable, and after mlkv_clear_status the same keys insert as if the failed
call had never been made.
"""
import ctypes
import time

import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import assert_bits, dev, host, torch_cuda

pytestmark = pytest.mark.gpu


def _lib():
    from paper_2504_01506_gb300 import _lib

    return _lib, _lib.load()


def _config(L, tiered=False):
    return L.Config(dim=16, insert_on_miss=1, capacity=20_000, max_batch=4_096, lr=0.1, eps=1e-8, state_init=0.0,
                    init_lo=-0.01, init_hi=0.01, seed=3, staleness_bound=0,
                    hbm_cache_rows=2 * 4_096 + 64 if tiered else 0, flags=0, reserved=0)


def _free_bytes(torch):
    torch.cuda.synchronize()
    free, _ = torch.cuda.mem_get_info()
    return free


@pytest.mark.parametrize("tiered", [False, True])
def test_every_allocation_of_open_failed_in_turn(tiered):
    torch = torch_cuda()
    L, lib = _lib()
    cfg = _config(L, tiered)
    # a first open and close, so that lazily created driver state is not counted
    h = ctypes.c_void_p()
    assert lib.mlkv_open(ctypes.byref(cfg), ctypes.byref(h)) == L.OK
    assert lib.mlkv_close(h) == L.OK
    base = _free_bytes(torch)
    failed = 0
    for nth in range(1, 64):
        assert lib.mlkv_debug_fail(L.FAULT_ALLOC, nth) == L.OK
        h = ctypes.c_void_p()
        rc = lib.mlkv_open(ctypes.byref(cfg), ctypes.byref(h))
        lib.mlkv_debug_fail(L.FAULT_ALLOC, 0)
        if rc == L.OK:  # nth is past the last allocation of open: the injection never fired
            assert h.value
            assert lib.mlkv_close(h) == L.OK
            break
        assert rc == L.ERR_NOMEM, (nth, rc)
        assert not h.value, nth
        assert _free_bytes(torch) == base, f"device memory left behind when allocation {nth} failed"
        failed += 1
    else:
        pytest.fail("open never succeeded")
    assert failed >= (12 if tiered else 5)  # every allocation of open was failed once
    assert _free_bytes(torch) == base


def _store_and_oracle(extra_capacity=0):
    from paper_2504_01506_gb300 import EmbeddingStore

    cfg = W.scaled(W.tiny(), 50, 4)
    store = EmbeddingStore(dim=cfg.dim, capacity=cfg.n_keys + extra_capacity, max_batch=max(cfg.batch, cfg.n_keys),
                           lr=cfg.lr,
                           eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi, seed=cfg.seed,
                           device="cuda:0")
    ref = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                       init_hi=cfg.init_hi, seed=cfg.seed, precision=32)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    ref.insert(pre)
    return cfg, store, ref, pre


def test_failed_staging_allocation_and_copies_leave_the_table_usable():
    torch = torch_cuda()
    from paper_2504_01506_gb300.store import MLKVError

    L, lib = _lib()
    cfg, store, ref, pre = _store_and_oracle()
    keys = cfg.batch_keys(0)
    grads = cfg.grads(0)
    hk = torch.from_numpy(keys).pin_memory()
    hg = torch.from_numpy(grads).pin_memory()
    hout = torch.empty((len(keys), cfg.dim), dtype=torch.float32).pin_memory()
    before_w, before_G = (host(x) for x in store.export(dev(pre)))

    # the first host-buffer call allocates its staging: fail the second of its two allocations
    lib.mlkv_debug_fail(L.FAULT_ALLOC, 2)
    with pytest.raises(MLKVError) as e:
        store.apply_grad_host(hk, hg)
    lib.mlkv_debug_fail(L.FAULT_ALLOC, 0)
    assert e.value.code == L.ERR_NOMEM
    # the key copy, then the gradient copy of an apply, each failed in turn
    for nth in (1, 2):
        lib.mlkv_debug_fail(L.FAULT_COPY, nth)
        with pytest.raises(MLKVError) as e:
            store.apply_grad_host(hk, hg)
        lib.mlkv_debug_fail(L.FAULT_COPY, 0)
        assert e.value.code == L.ERR_CUDA
    # the Get's output copy back failed
    lib.mlkv_debug_fail(L.FAULT_COPY, 2)
    with pytest.raises(MLKVError) as e:
        store.get_host(hk, hout)
    lib.mlkv_debug_fail(L.FAULT_COPY, 0)
    assert e.value.code == L.ERR_CUDA
    assert store.sync() == 0
    # nothing was applied
    w, G = (host(x) for x in store.export(dev(pre)))
    assert_bits(w, before_w, "rows after the failed applies")
    assert_bits(G, before_G, "state after the failed applies")

    # the table still works, through host buffers, against the oracle
    store.get_host(hk, hout)
    store.apply_grad_host(hk, hg)
    torch.cuda.synchronize()
    assert store.sync() == 0
    want, _, _ = ref.get(keys)
    assert_bits(hout.numpy(), want, "Get through host buffers after the failures")
    ref.apply_grad(keys, grads)
    u = np.unique(keys)
    w, G = store.export(dev(u))
    rw, rG = ref.export(u)
    # the tiny workload's short runs are summed in occurrence order: bit-exact
    counts = np.unique(keys, return_counts=True)[1]
    short = counts <= 32
    assert_bits(host(w)[short], rw[short], "rows after a good apply")
    assert_bits(host(G)[short], rG[short], "state after a good apply")
    store.close()


def test_wait_that_runs_out_reports_timeout():
    torch = torch_cuda()
    L, lib = _lib()
    cfg, store, ref, pre = _store_and_oracle(extra_capacity=1000)
    new = (np.arange(600, dtype=np.int64) * 7919 + (1 << 45))[np.random.default_rng(3).permutation(600)]
    new = np.concatenate([new, new[:100]])  # duplicates: first occurrences decide the row ids
    lib.mlkv_debug_fail(L.FAULT_WAIT, 1)  # the next launch of the miss kernel
    t0 = time.time()
    store.insert(dev(new))
    rc = store.sync()
    took = time.time() - t0
    lib.mlkv_debug_fail(L.FAULT_WAIT, 0)
    assert rc == L.ERR_TIMEOUT, rc
    assert took < 60, took
    assert store.size() == len(pre)  # no row handed out
    store.clear_status()
    assert store.sync() == 0
    # the context and the table work: the same keys insert as if the failed call never ran
    store.insert(dev(new))
    assert store.sync() == 0
    ref.insert(new)
    assert store.size() == len(pre) + 600 == ref.size()
    assert np.array_equal(host(store.find(dev(new))), ref.find(new))
    got = host(store.get(dev(new)))
    want, _, _ = ref.get(new)
    assert_bits(got, want, "Get of the keys after the timed-out insert")
    store.close()


def test_apply_whose_miss_wait_runs_out_updates_only_known_keys():
    """An apply with new keys whose miss kernel gives up: the new keys get no
    rows, the sort still sees every lookup (its first pass is counted by the
    probe and the miss kernel), the known keys are updated as if the new keys'
    lookups were not in the batch, and the status is MLKV_ERR_TIMEOUT."""
    torch = torch_cuda()
    L, lib = _lib()
    cfg, store, ref, pre = _store_and_oracle(extra_capacity=2000)
    keys = cfg.batch_keys(0).copy()
    grads = cfg.grads(0)
    rng = np.random.default_rng(11)
    new = (np.arange(len(keys) // 8, dtype=np.int64) * 104729 + (1 << 46))
    at = rng.choice(len(keys), size=len(keys) // 4, replace=False)
    keys[at] = new[rng.integers(0, len(new), size=len(at))]  # new keys, some repeated
    known = ~np.isin(keys, new)
    lib.mlkv_debug_fail(L.FAULT_WAIT, 1)  # the apply's miss kernel
    t0 = time.time()
    store.apply_grad(dev(keys), dev(grads))
    rc = store.sync()
    took = time.time() - t0
    lib.mlkv_debug_fail(L.FAULT_WAIT, 0)
    assert rc == L.ERR_TIMEOUT, rc
    assert took < 60, took
    store.clear_status()
    assert store.sync() == 0
    assert store.size() == len(pre)  # no new key got a row
    ref.apply_grad(keys[known], grads[known])
    u, c = np.unique(keys[known], return_counts=True)
    w, G = store.export(dev(u))
    rw, rG = ref.export(u)
    short = c <= 32
    assert short.sum() > 100
    assert_bits(host(w)[short], rw[short], "known keys' rows after the timed-out apply")
    assert_bits(host(G)[short], rG[short], "known keys' state after the timed-out apply")
    # the same apply again inserts the new keys and updates everything
    store.apply_grad(dev(keys), dev(grads))
    assert store.sync() == 0
    ref.apply_grad(keys, grads)
    assert store.size() == ref.size() == len(pre) + len(np.unique(keys[~known]))
    u, c = np.unique(keys, return_counts=True)
    w, G = store.export(dev(u))
    rw, rG = ref.export(u)
    short = c <= 32
    assert_bits(host(w)[short], rw[short], "rows after the second apply")
    assert_bits(host(G)[short], rG[short], "state after the second apply")
    store.close()

"""Pins of the oracle to facts that do not come from the oracle itself.

Each check takes the oracle's ctypes library (the real build, or a build with
one planted mistake) and raises AssertionError when the oracle disagrees with
a published test vector, a closed form, a brute-force recount, an invariant or
a hand-worked value.  ``test_oracle_pins.py`` runs them on the real oracle;
``test_oracle_mutants.py`` shows that every planted mistake fails at least one.
"""
import math
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
F32_ULP = 2.0 ** -23


def _ulp(x: float) -> float:
    return float(np.spacing(np.float32(abs(x)))) if x != 0 else float(np.finfo(np.float32).tiny)


def _table(lib, dim, **kw):
    return oracle.Table(dim, lib=lib, **kw)


# --- counter-based init ---------------------------------------------------------

def check_splitmix64_vectors(lib):
    """Published SplitMix64 outputs from state 0 (tests/golden/splitmix64_vectors.txt)."""
    with open(os.path.join(GOLDEN, "splitmix64_vectors.txt")) as f:
        rows = [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]
    assert rows
    for _, state, out in rows:
        assert oracle.splitmix64(int(state, 16), lib=lib) == int(out, 16)


def check_init_lattice_and_range(lib):
    """init(0,1) values lie on the 2^-24 lattice in [0,1); init(lo,hi) lies in
    [lo,hi) and is the affine image of init(0,1); values look uniform."""
    seed = 12345
    keys = [0, 1, 2, 3, 2**40 - 1, 2**63 + 5, 7 << 32]
    u = np.array([[oracle.init_value(seed, k, j, 0.0, 1.0, lib=lib) for j in range(64)] for k in keys])
    assert np.all((u >= 0) & (u < 1))
    scaled = u * 2.0**24
    assert np.all(scaled == np.floor(scaled))
    lo, hi = -0.01, 0.01
    v = np.array([[oracle.init_value(seed, k, j, lo, hi, lib=lib) for j in range(64)] for k in keys])
    assert np.all((v >= np.float32(lo)) & (v < np.float32(hi)))
    span = np.float32(hi) - np.float32(lo)
    expect = np.float32(lo) + (u.astype(np.float32) * span)
    assert np.all(np.abs(v - expect) <= np.spacing(np.float32(0.01)) * 2)
    # uniformity: 4,096 draws in 16 bins, chi-square well below the 1e-4 tail (~ 43)
    draws = np.array([oracle.init_value(seed, k, j, 0.0, 1.0, lib=lib)
                      for k in range(256) for j in range(16)])
    hist = np.histogram(draws, bins=16, range=(0, 1))[0]
    chi2 = float(((hist - 256.0) ** 2 / 256.0).sum())
    assert chi2 < 43.0, chi2
    assert abs(draws.mean() - 0.5) < 0.03


def check_init_is_counter_based(lib):
    """A key's init row does not depend on when or where it is inserted."""
    a = _table(lib, 8, seed=99)
    b = _table(lib, 8, seed=99)
    a.insert([5, 6, 7])
    b.insert([7, 100, 200, 5])
    wa, _ = a.export([5, 7])
    wb, _ = b.export([5, 7])
    assert np.array_equal(wa.view(np.uint32), wb.view(np.uint32))
    want = np.array([[oracle.init_value(99, k, j, -0.01, 0.01, lib=lib) for j in range(8)] for k in (5, 7)],
                    np.float32)
    assert np.array_equal(wa.view(np.uint32), want.view(np.uint32))
    c = _table(lib, 8, seed=100)
    c.insert([5])
    assert not np.array_equal(c.export([5])[0], wa[:1])


# --- Adagrad closed forms ---------------------------------------------------------

def check_adagrad_eps0_constant_gradient(lib):
    """eps = 0, G0 = 0, gradient c every step: G_k = k c^2 and
    w_k = w0 - lr sign(c) * sum_{i<=k} 1/sqrt(i) (generalised harmonic number)."""
    lr, c, steps = 0.05, 0.5, 40
    t = _table(lib, 2, lr=lr, eps=0.0)
    w0 = np.array([[0.25, -0.75]], np.float32)
    t.put([1], w0)
    for k in range(1, steps + 1):
        t.apply_grad([1], np.array([[c, -c]], np.float32))
        w, G = t.export([1])
        assert G[0, 0] == k * c * c and G[0, 1] == k * c * c
        h = math.fsum(1.0 / math.sqrt(i) for i in range(1, k + 1))
        assert abs(w[0, 0] - (0.25 - lr * h)) <= 8 * k * F32_ULP
        assert abs(w[0, 1] - (-0.75 + lr * h)) <= 8 * k * F32_ULP


def check_adagrad_scale_invariance(lib):
    """eps = 0: scaling every gradient by 2^m leaves the rows bit-identical and
    scales the state by exactly 4^m (every step is exact under 2^m scaling)."""
    rng = np.random.default_rng(3)
    keys = rng.integers(0, 6, 200)
    g = rng.standard_normal((200, 4)).astype(np.float32)
    a = _table(lib, 4, lr=0.1, eps=0.0, seed=4)
    b = _table(lib, 4, lr=0.1, eps=0.0, seed=4)
    for s in range(0, 200, 50):
        a.apply_grad(keys[s:s + 50], g[s:s + 50])
        b.apply_grad(keys[s:s + 50], g[s:s + 50] * np.float32(32.0))
    wa, Ga = a.export(np.arange(6))
    wb, Gb = b.export(np.arange(6))
    assert np.array_equal(wa.view(np.uint32), wb.view(np.uint32))
    assert np.array_equal(Ga * np.float32(1024.0), Gb)


def check_adagrad_eps_placement(lib):
    """One step from G0 = 0 with g = eps: g / (sqrt(g^2) + eps) = 1/2 exactly
    (dyadic values, so every fp32 operation is exact)."""
    eps = 2.0 ** -10
    lr = 0.25
    t = _table(lib, 1, lr=lr, eps=eps)
    t.put([3], np.array([[1.0]], np.float32))
    t.apply_grad([3], np.array([[eps]], np.float32))
    w, G = t.export([3])
    assert G[0, 0] == eps * eps
    assert w[0, 0] == 1.0 - lr / 2


def check_adagrad_state_init(lib):
    """state_init = 3 g^2, eps = 0: G = 4 g^2, step = lr/2 (all exact)."""
    g = 0.125
    t = _table(lib, 1, lr=0.5, eps=0.0, state_init=3 * g * g)
    t.put([9], np.array([[0.75]], np.float32))
    _, G0 = t.export([9])
    assert G0[0, 0] == 3 * g * g
    t.apply_grad([9], np.array([[g]], np.float32))
    w, G = t.export([9])
    assert G[0, 0] == 4 * g * g
    assert w[0, 0] == np.float32(0.75) - np.float32(0.25)


def check_duplicates_one_step_on_sum(lib):
    """Duplicate keys in one apply batch: one step on the summed gradient.
    eps = 0 and dyadic gradients: G = (sum)^2 and the step is lr * sign(sum)."""
    t = _table(lib, 1, lr=0.5, eps=0.0)
    t.put([4], np.array([[2.0]], np.float32))
    t.apply_grad([4, 4, 4], np.array([[0.25], [0.5], [-0.125]], np.float32))
    w, G = t.export([4])
    assert G[0, 0] == 0.625 ** 2
    assert w[0, 0] == 1.5
    # interleaved keys: each distinct key equals a single occurrence carrying the
    # fp32 occurrence-order sum of its gradients
    rng = np.random.default_rng(5)
    keys = np.array([1, 2, 1, 3, 1, 2, 4, 1])
    g = rng.standard_normal((8, 3)).astype(np.float32)
    a = _table(lib, 3, lr=0.1, eps=1e-8, seed=6)
    a.apply_grad(keys, g)
    for k in (1, 2, 3, 4):
        s = np.zeros(3, np.float32)
        for i in np.nonzero(keys == k)[0]:
            s = s + g[i]
        b = _table(lib, 3, lr=0.1, eps=1e-8, seed=6)
        b.apply_grad([k], s[None, :])
        wa, Ga = a.export([k])
        wb, Gb = b.export([k])
        assert np.array_equal(wa.view(np.uint32), wb.view(np.uint32))
        assert np.array_equal(Ga.view(np.uint32), Gb.view(np.uint32))


def check_zero_gradient_and_columns(lib):
    """A zero gradient changes nothing; a gradient in one column leaves the
    other columns bit-identical."""
    t = _table(lib, 4, lr=0.1, eps=1e-8, state_init=0.5, seed=8)
    t.insert([11])
    w0, G0 = t.export([11])
    t.apply_grad([11], np.zeros((1, 4), np.float32))
    w1, G1 = t.export([11])
    assert np.array_equal(w0, w1) and np.array_equal(G0, G1)
    t.apply_grad([11], np.array([[0.0, 0.0, 0.3, 0.0]], np.float32))
    w2, G2 = t.export([11])
    for j in (0, 1, 3):
        assert w2[0, j] == w0[0, j] and G2[0, j] == G0[0, j]
    assert w2[0, 2] < w0[0, 2] and G2[0, 2] > G0[0, 2]


def check_adagrad_hand_values(lib):
    """Hand-worked single-key steps (tests/golden/adagrad_hand.txt)."""
    with open(os.path.join(GOLDEN, "adagrad_hand.txt")) as f:
        lines = [ln for ln in f if ln.strip() and not ln.startswith("#")]
    assert lines
    for ln in lines:
        head, grads, tail = ln.split("|")
        lr, eps, s0, w0 = map(float, head.split())
        gs = [float(x) for x in grads.split()]
        G_want, w_want = map(float, tail.split())
        t = _table(lib, 1, lr=lr, eps=eps, state_init=s0)
        t.put([1], np.array([[w0]], np.float32))
        for g in gs:
            t.apply_grad([1], np.array([[g]], np.float32))
        w, G = t.export([1])
        assert abs(float(G[0, 0]) - G_want) <= 4 * _ulp(G_want), (ln, G)
        assert abs(float(w[0, 0]) - w_want) <= 6 * _ulp(w_want), (ln, w)


# --- dedup and segment sums: brute force -------------------------------------------

def check_dedup_bruteforce(lib):
    rng = np.random.default_rng(11)
    for n, pool in ((1, 1), (7, 3), (120, 10), (300, 1000), (64, 1)):
        keys = rng.integers(0, pool, n) * 1_000_003 + 17
        uniq, counts, first = oracle.dedup(keys, lib=lib)
        # O(n^2): the first occurrence of each distinct key, in position order
        want_first = [i for i in range(n) if all(keys[j] != keys[i] for j in range(i))]
        assert list(first) == want_first
        assert list(uniq) == [int(keys[i]) for i in want_first]
        assert list(counts) == [sum(int(keys[j] == keys[i]) for j in range(n)) for i in want_first]
        assert counts.sum() == n


def check_segment_sums_bruteforce(lib):
    """fp32 occurrence-order sums lie within the recursive-summation bound
    (n-1) u sum|g| of the exactly rounded sum (math.fsum); fp64 sums within
    fp32 rounding of it."""
    rng = np.random.default_rng(12)
    n, d = 400, 5
    keys = rng.integers(0, 7, n)
    g = (rng.standard_normal((n, d)) * 0.01).astype(np.float32)
    for prec in (32, 64):
        uniq, sums = oracle.segment_sums(keys, g, d, precision=prec, lib=lib)
        assert sorted(uniq.tolist()) == sorted(set(keys.tolist()))
        for u, k in enumerate(uniq):
            idx = np.nonzero(keys == k)[0]
            for j in range(d):
                exact = math.fsum(float(g[i, j]) for i in idx)
                mag = math.fsum(abs(float(g[i, j])) for i in idx)
                bound = (len(idx) * 2.0 ** -24) * mag if prec == 32 else 2.0 ** -24 * abs(exact) + 1e-30
                assert abs(float(sums[u, j]) - exact) <= bound + 1e-45, (prec, k, j)


# --- key -> row, Get / Put ------------------------------------------------------------

def check_row_alloc_golden(lib):
    """Hand-worked row ids under first-occurrence allocation (tests/golden/row_alloc.txt)."""
    with open(os.path.join(GOLDEN, "row_alloc.txt")) as f:
        lines = [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]
    t = _table(lib, 2, seed=1)
    for ln in lines:
        lhs, rhs = ln.split("->")
        op, *ks = lhs.split()
        keys = np.array([int(x) for x in ks], np.int64)
        want = [int(x) for x in rhs.split()]
        if op == "size":
            assert t.size() == want[0], ln
            continue
        if op == "insert":
            t.insert(keys)
        elif op == "get":
            t.get(keys)
        elif op == "put":
            t.put(keys, np.ones((len(keys), 2), np.float32))
        elif op == "apply":
            t.apply_grad(keys, np.ones((len(keys), 2), np.float32))
        assert t.find(keys).tolist() == want, ln


def check_get_put_semantics(lib):
    d = 6
    t = _table(lib, d, seed=21, state_init=0.25)
    rng = np.random.default_rng(13)
    keys = np.array([5, 9, 5, 12], np.int64)
    vals = rng.standard_normal((4, d)).astype(np.float32)
    t.insert([9])
    _, G9 = t.export([9])
    t.put(keys, vals)
    out, rows, rc = t.get([5, 9, 12])
    assert rc == oracle.OK
    # Get after Put returns the Put value bit-exactly; the later duplicate wins
    assert np.array_equal(out[0].view(np.uint32), vals[2].view(np.uint32))
    assert np.array_equal(out[1].view(np.uint32), vals[1].view(np.uint32))
    assert np.array_equal(out[2].view(np.uint32), vals[3].view(np.uint32))
    # Put keeps the state of a present key and gives new keys state_init
    _, G = t.export([9, 5, 12])
    assert np.array_equal(G[0], G9[0]) and np.all(G[1:] == np.float32(0.25))
    # Get of an untouched key inserts it with the init row
    out2, rows2, _ = t.get([77])
    want = [oracle.init_value(21, 77, j, -0.01, 0.01, lib=lib) for j in range(d)]
    assert np.array_equal(out2[0], np.array(want, np.float32))
    assert t.size() == 4 and len(set(t.find([5, 9, 12, 77]).tolist())) == 4
    # without insert-on-miss: NaN, NOT_FOUND, nothing inserted
    s = _table(lib, d, seed=21, insert_on_miss=False)
    s.insert([1])
    o, r, rc = s.get([1, 2])
    assert rc == oracle.NOT_FOUND and r.tolist() == [0, -1]
    assert np.all(np.isnan(o[1])) and not np.any(np.isnan(o[0]))
    assert s.apply_grad([2, 1], np.ones((2, d), np.float32)) == oracle.NOT_FOUND
    assert s.size() == 1
    w1, _ = s.export([1])
    assert np.all(w1 < o[0])  # the present key was still updated


def check_precisions_agree(lib):
    """fp32 op-by-op and fp64 evaluation agree to fp32 accuracy on a random run."""
    rng = np.random.default_rng(14)
    a = _table(lib, 8, lr=0.1, seed=2, precision=32)
    b = _table(lib, 8, lr=0.1, seed=2, precision=64)
    for _ in range(5):
        keys = rng.integers(0, 50, 300)
        g = (rng.standard_normal((300, 8)) * 0.01).astype(np.float32)
        a.apply_grad(keys, g)
        b.apply_grad(keys, g)
    wa, Ga = a.export(np.arange(50))
    wb, Gb = b.export(np.arange(50))
    assert np.all(np.abs(wa - wb) <= 1e-5 * (1 + np.abs(wb)))
    assert np.all(np.abs(Ga - Gb) <= 1e-5 * (1 + np.abs(Gb)))


def check_import_semantics(lib):
    """Import is an upsert of row and state: what was imported comes back out,
    the later duplicate wins, no state keeps the current one (state_init for a
    new key), and new keys get the next row ids in order."""
    d = 5
    t = _table(lib, d, seed=3, state_init=0.5)
    t.insert([40, 41])
    rng = np.random.default_rng(15)
    rows = rng.standard_normal((4, d)).astype(np.float32)
    state = np.abs(rng.standard_normal((4, d))).astype(np.float32)
    assert t.import_([41, 50, 41, 60], rows, state) == oracle.OK
    w, G = t.export([41, 50, 60])
    for got, want in ((w[0], rows[2]), (w[1], rows[1]), (w[2], rows[3]),
                      (G[0], state[2]), (G[1], state[1]), (G[2], state[3])):
        assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    assert t.keys().tolist() == [40, 41, 50, 60] and t.find([50, 60]).tolist() == [2, 3]
    _, G40 = t.export([40])
    t.import_([40, 70], rows[:2])  # no state
    _, G2 = t.export([40, 70])
    assert np.array_equal(G2[0], G40[0]) and np.all(G2[1] == np.float32(0.5))


def check_checkpoint_resume(lib):
    """A table restored from its keys (row order), rows and state has the same
    row ids and continues bit-identically with the original."""
    d = 4
    kw = dict(lr=0.1, seed=8, state_init=0.0)
    a = _table(lib, d, **kw)
    rng = np.random.default_rng(16)
    batches = [(rng.integers(0, 300, 200), (rng.standard_normal((200, d)) * 0.1).astype(np.float32))
               for _ in range(6)]
    for k, g in batches[:3]:
        a.get(k)
        a.apply_grad(k, g)
    keys = a.keys()
    w, G = a.export(keys)
    b = _table(lib, d, **kw)
    b.import_(keys, w, G)
    assert np.array_equal(b.find(keys), np.arange(len(keys)))
    for k, g in batches[3:]:
        oa, _, _ = a.get(k)
        ob, _, _ = b.get(k)
        assert np.array_equal(oa.view(np.uint32), ob.view(np.uint32))
        a.apply_grad(k, g)
        b.apply_grad(k, g)
    wa, Ga = a.export(a.keys())
    wb, Gb = b.export(a.keys())
    assert np.array_equal(wa.view(np.uint32), wb.view(np.uint32))
    assert np.array_equal(Ga.view(np.uint32), Gb.view(np.uint32))


ALL_CHECKS = [v for k, v in sorted(globals().items()) if k.startswith("check_")]

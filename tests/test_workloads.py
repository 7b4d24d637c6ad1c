"""The seeded input generators: Zipf law, bijections, config shapes, determinism."""
import math

import numpy as np
import pytest

import workloads as W
from workloads.zipf import ZipfSampler, scatter_bijection


@pytest.mark.parametrize("alpha", [0.5, 0.9, 1.0, 1.05, 1.2])
def test_zipf_chi_square(alpha):
    n, m = 40, 400_000
    z = ZipfSampler(n, alpha)
    x = z.sample(np.random.default_rng(1), m)
    assert x.min() >= 1 and x.max() <= n
    obs = np.bincount(x, minlength=n + 1)[1:]
    exp = z.pmf(np.arange(1, n + 1)) * m
    chi2 = float(((obs - exp) ** 2 / exp).sum())
    # 39 degrees of freedom: the 1e-4 upper tail is ~ 80
    assert chi2 < 80.0, chi2


def test_zipf_expected_unique():
    n, b, trials = 5_000, 2_000, 20
    z = ZipfSampler(n, 1.1)
    p = z.pmf(np.arange(1, n + 1))
    want = float(np.sum(1.0 - (1.0 - p) ** b))
    rng = np.random.default_rng(2)
    got = np.mean([len(np.unique(z.sample(rng, b))) for _ in range(trials)])
    assert abs(got - want) < 0.02 * want


def test_zipf_large_n_head():
    n = 4_000_000
    z = ZipfSampler(n, 1.2)
    x = z.sample(np.random.default_rng(3), 400_000)
    h = math.fsum(k ** -1.2 for k in range(1, 200_001)) + (200_000.5 ** -0.2 - (n + 0.5) ** -0.2) / 0.2
    p1 = 1.0 / h
    assert abs(np.mean(x == 1) - p1) < 5 * math.sqrt(p1 * (1 - p1) / len(x))


@pytest.mark.parametrize("n", [1, 2, 1000, 4_000_000, 10_007])
def test_bijection_is_permutation(n):
    f = scatter_bijection(n, np.random.default_rng(n))
    m = min(n, 200_000)
    r = np.arange(1, m + 1)
    out = f(r)
    assert out.min() >= 0 and out.max() < n
    assert len(np.unique(out)) == m


def test_tiny_config():
    c = W.tiny()
    keys = c.preload_keys()
    assert len(keys) == 100_000 and len(np.unique(keys)) == 100_000
    assert keys.min() >= 0 and keys.max() < 2**40
    b = c.batch_keys(0)
    assert len(b) == 4_096 and np.all(np.isin(b, keys))
    assert np.array_equal(b, W.tiny().batch_keys(0))
    assert not np.array_equal(b, c.batch_keys(1))
    g = c.grads(0)
    assert g.shape == (4_096, 16) and g.dtype == np.float32
    assert abs(float(g.std()) - 0.01) < 5e-4


def test_dlrm_config_shape():
    c = W.scaled(W.dlrm(), 100, 64)
    b = c.batch_keys(0)
    assert len(b) == c.batch and c.batch % 26 == 0
    t, r = b >> 32, b & 0xFFFFFFFF
    assert np.all(t == np.tile(np.arange(26), c.batch // 26))
    assert r.max() < c.rows_per_table
    pre = c.preload_keys()
    assert len(pre) == c.n_keys and np.all(np.isin(b, pre))


def test_kg_config_shape():
    c = W.scaled(W.kg(), 1000, 10)
    b = c.batch_keys(0)
    assert len(b) == c.batch
    rel = b >= W.RELATION_BASE
    assert rel.sum() == c.triples
    assert np.all(b[~rel] < c.entities) and np.all(b[rel] - W.RELATION_BASE < c.relations)
    assert np.all(np.isin(b, c.preload_keys()))


def test_gnn_config_shape():
    c = W.scaled(W.gnn(), 1000, 64)
    b = c.batch_keys(0)
    assert len(b) == c.seeds * 261
    assert b.min() >= 0 and b.max() < c.nodes
    # hop samples are heavy-tailed: far fewer distinct keys than lookups
    assert len(np.unique(b[c.seeds:])) < 0.8 * (len(b) - c.seeds)


def test_full_size_batches():
    for name, want in (("dlrm", 1_703_936), ("kg", 200_000), ("tiered", 1_048_576)):
        c = W.ALL[name]()
        b = c.batch_keys(0)
        assert len(b) == want == c.batch


@pytest.mark.parametrize("make", [W.ycsb, W.ycsb_uniform])
def test_ycsb_batches(make):
    """A YCSB-shaped batch: 1,048,576 operations over 50M records of 256 fp32,
    each a Get or a Put by a fair coin (the 50/50 mix), written values
    N(0, 0.01); keys Zipf(0.99) scattered over the records, or uniform."""
    c = W.scaled(make(), 50, 8)  # 1M records, batches of 131,072: the same distributions
    r, w, v = c.ops(0)
    n = len(r) + len(w)
    assert n == c.batch
    assert abs(len(r) / n - 0.5) < 4 * math.sqrt(0.25 / n)
    assert v.shape == (len(w), 256) and v.dtype == np.float32
    assert abs(float(v.std()) - 0.01) < 1e-4 and abs(float(v.mean())) < 1e-4
    keys = np.concatenate([r, w])
    assert keys.min() >= 0 and keys.max() < c.n_keys
    _, counts = np.unique(keys, return_counts=True)
    if c.alpha:
        # Zipf(0.99) over N records: the hottest key takes 1 / H(N, 0.99) of the lookups
        want = 1.0 / float(np.sum(np.arange(1, c.n_keys + 1, dtype=np.float64) ** -0.99))
        assert abs(counts.max() / n - want) < 0.1 * want
    else:
        assert counts.max() < 10  # uniform over 1M records: no hot key
    r2, w2, v2 = c.ops(0)
    assert np.array_equal(r, r2) and np.array_equal(w, w2) and np.array_equal(v, v2)  # seeded

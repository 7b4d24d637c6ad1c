"""The dedup sort on every path it takes: one, two and four radix passes (the
row-id bits follow the capacity), tiles of 1,024 and of 4,096 lookups (batches
on both sides of 2^19, with ragged last tiles), the first pass counted by the
apply's probe or by the histogram kernel (dedup), and the later passes counted
by the scatter before them, with gradient applies and dedups alternating so
that a count or total left behind by one sort would corrupt the next.

The gradients are small multiples of 2^-10, so every run's sum is exact in fp32
whatever the order it is added in: the rows and states of every key, long runs
included, must then equal the oracle's fp32 op-by-op values bit for bit, and a
lookup sorted into the wrong run shows as a wrong sum."""
import numpy as np
import pytest

import oracle
import workloads as W
from gpu_helpers import assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu

SMALL = 1 << 19  # batches below this sort in tiles of 1,024 lookups
SIZES = [3 * 1024 + 5, SMALL - 1, SMALL, SMALL + 4096 + 7, 1]


@pytest.mark.parametrize("capacity,passes", [(300, 1), (20_000, 2), (1 << 28, 4)])
def test_sort_paths_exact_sums(capacity, passes):
    torch_cuda()
    cfg = W.tiny()
    cfg.dim = 1 if capacity > 1_000_000 else 4
    n_keys = min(capacity - 10, 50_000)
    store, ref = make_pair(cfg, capacity=capacity, max_batch=max(SIZES), lr=0.125, eps=1e-8)
    rng = np.random.default_rng(passes)
    universe = rng.choice(1 << 40, n_keys, replace=False).astype(np.int64)
    store.insert(dev(universe))
    ref.insert(universe)
    weights = 1.0 / np.arange(1, n_keys + 1) ** 1.1
    weights /= weights.sum()
    # bits of a row id (the sentinel of a lookup without a row included), the
    # digits of at most 9 bits spread over the fewest passes
    bits = int(capacity).bit_length()
    assert -(-bits // 9) == passes
    seen = set()
    for i, n in enumerate(SIZES):
        keys = universe[rng.choice(n_keys, n, p=weights)]
        grads = (rng.integers(-8, 9, size=(n, cfg.dim)) * 2.0**-10).astype(np.float32)
        store.get(dev(keys))
        ref.get(keys)
        store.apply_grad(dev(keys), dev(grads))
        ref.apply_grad(keys, grads)
        assert store.last_unique() == len(np.unique(keys)), f"distinct rows, batch of {n}"
        seen.update(keys.tolist())
        # a dedup of another batch, then the next apply
        dk = universe[rng.choice(n_keys, SIZES[(i + 2) % len(SIZES)], p=weights)]
        uniq, counts = store.dedup(dev(dk))
        uniq, counts = host(uniq), host(counts)
        ou, oc, _ = oracle.dedup(dk)
        o, g = np.argsort(ou), np.argsort(uniq)
        assert np.array_equal(uniq[g], ou[o]), f"dedup keys, batch of {len(dk)}"
        assert np.array_equal(counts[g].astype(np.int64), oc[o]), f"dedup counts, batch of {len(dk)}"
    touched = np.array(sorted(seen), dtype=np.int64)
    w, G = store.export(dev(touched))
    rw, rG = ref.export(touched)
    assert store.sync() == 0
    assert_bits(host(w), rw, "rows")
    assert_bits(host(G), rG, "state")

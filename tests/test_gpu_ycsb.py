"""YCSB-shaped batches of Gets and Puts (MLKV Section 4.5: 50% reads, 50%
writes, uniform or skewed keys) against the oracle: a batch's Gets read the
records as they were before the batch, then its Puts write them (the later of
two Puts of a key wins).  Gets and the final records are bit-exact."""
import numpy as np
import pytest

import workloads as W
from gpu_helpers import assert_bits, dev, host, make_pair, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("make", [W.ycsb, W.ycsb_uniform])
def test_get_put_batches_match_the_oracle(make):
    torch_cuda()
    cfg = W.scaled(make(), 1_000, 100)  # 50,000 records of 256 fp32, batches of 10,485 operations
    store, ref = make_pair(cfg, max_batch=cfg.n_keys)
    pre = cfg.preload_keys()
    store.insert(dev(pre))
    ref.insert(pre)
    for step in range(5):
        r, w, v = cfg.ops(step)
        assert_bits(host(store.get(dev(r))), ref.get(r)[0], f"Get, step {step}")
        store.put(dev(w), dev(v))
        ref.put(w, v)
    assert store.sync() == 0
    w_all, G_all = store.export(dev(pre))
    rw, rG = ref.export(pre)
    assert_bits(host(w_all), rw, "records")
    assert_bits(host(G_all), rG, "state (Put keeps it)")

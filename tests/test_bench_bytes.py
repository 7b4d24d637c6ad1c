"""bench.py's algorithmic byte model (what roofline.achieved divides by), on a
batch whose runs are counted by hand, and the rule for its measured traffic.

Batch: key 7 once (a run of one lookup), key 5 twice and key 9 three times
(small runs: 2-4 lookups), key 11 six times (a short run of 5-32), key 3 forty
times (a long run: more than 32 lookups, one chunk of 64).  dim 4, so a row is
16 bytes."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

D = 4
ROW = 4 * D


def _batch():
    keys = np.array([7] + [5] * 2 + [9] * 3 + [11] * 6 + [3] * 40, np.int64)
    return np.random.default_rng(0).permutation(keys)


def test_run_split_of_the_batch():
    s = bench.batch_stats(_batch(), D)
    assert (s["B"], s["U"]) == (52, 5)
    assert (s["Bl"], s["Ul"], s["items"]) == (40, 1, 1)   # the long run: one chunk
    assert (s["Bs"], s["Us"]) == (12, 4)                  # the runs of up to 32, singletons included
    assert (s["U1"], s["Usm"], s["Bsm"]) == (1, 2, 5)     # key 7 alone; keys 5 and 9 small
    assert (s["Um"], s["Bs"] - s["U1"] - s["Bsm"]) == (1, 6)  # key 11: a short run of 6


def test_bytes_per_kernel():
    s = bench.batch_stats(_batch(), D)
    # Get: each lookup's key and output row; each distinct key's index sector and row
    assert bench.kernel_bytes(s, 1, 3) == 52 * (8 + ROW) + 5 * (32 + ROW)
    # k_single: the gradient row, row and state read and written, the 8-byte record
    assert bench.kernel_bytes(s, 10, 3) == 1 * (ROW + 4 * ROW + 8)
    # k_small: 5 lookups' gradient rows; 2 runs' row and state and 20-byte records
    assert bench.kernel_bytes(s, 11, 3) == 5 * ROW + 2 * (4 * ROW + 20)
    # k_short: 6 lookups' gradient rows and positions; 1 run's row and state and record
    assert bench.kernel_bytes(s, 4, 3) == 6 * (ROW + 4) + 1 * (4 * ROW + 16)
    # k_long_sum: 40 gradient rows and positions, one chunk sum written
    assert bench.kernel_bytes(s, 5, 3) == 40 * (ROW + 4) + 1 * ROW
    # k_long_combine: the chunk sum read, the long run's row and state read and written
    assert bench.kernel_bytes(s, 7, 3) == 1 * ROW + 1 * 4 * ROW
    # the sort's scatter pass: (row id, position) read and written per lookup
    assert bench.kernel_bytes(s, 3, 3) == 52 * 16
    # the whole step, what the method must move: B(16 + 8d) + U(32 + 20d)
    assert s["step"] == 52 * (16 + 8 * D) + 5 * (32 + 20 * D)


def test_every_row_byte_is_counted_once_across_the_reduce_kernels():
    """Gradient rows: every lookup's once (in k_single, k_small, k_short or
    k_long_sum); row and state read and written: every distinct key's once (in
    k_single, k_small, k_short or k_long_combine)."""
    s = bench.batch_stats(_batch(), D)
    grads = s["U1"] * ROW + s["Bsm"] * ROW + (s["Bs"] - s["U1"] - s["Bsm"]) * ROW + s["Bl"] * ROW
    assert grads == s["B"] * ROW
    rmw = (s["U1"] + s["Usm"] + s["Um"] + s["Ul"]) * 4 * ROW
    assert rmw == s["U"] * 4 * ROW


def test_traffic_figures_only_for_their_workload_and_source(tmp_path):
    """roofline.traffic comes from a committed ncu figure only when it was taken
    on the same workload (name, rows, batch) and the kernel's current source."""
    import hashlib
    import json

    import workloads as W

    src = os.path.join(ROOT, "paper_2504_01506_gb300", "csrc", bench.KERNEL_SOURCES[1])
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    dlrm = W.dlrm()
    rec = {"workload": "dlrm", "rows": dlrm.n_keys, "batch_lookups": dlrm.batch, "bytes_per_launch": 123.0,
           "source_sha": sha}
    path = tmp_path / "traffic.json"
    path.write_text(json.dumps({"1": rec}))
    assert bench.traffic_for(1, dlrm, str(path)) == 123.0
    assert bench.traffic_for(1, W.kg(), str(path)) is None                     # another workload
    assert bench.traffic_for(1, W.scaled(dlrm, 10, 1), str(path)) is None      # same name, smaller table
    assert bench.traffic_for(2, dlrm, str(path)) is None                       # no figure for the kernel
    path.write_text(json.dumps({"1": dict(rec, source_sha="0" * 16)}))
    assert bench.traffic_for(1, dlrm, str(path)) is None                       # kernel source changed since

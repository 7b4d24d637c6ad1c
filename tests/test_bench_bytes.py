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
    on the same workload and batch size and on the kernel's current source; it
    is scaled to the launch by the algorithmic bytes."""
    import json

    import workloads as W

    dlrm = W.dlrm()
    rec = {"rows": dlrm.n_keys // 26, "scale": 26, "batch_lookups": dlrm.batch, "bytes_per_launch": 120.0,
           "algorithmic_bytes_per_launch": 100.0, "source_sha": bench.source_sha(1)}
    path = tmp_path / "traffic.json"
    path.write_text(json.dumps({"dlrm": {"1": rec}}))
    assert bench.traffic_for(1, dlrm, 200.0, str(path)) == 240.0               # scaled by the algorithmic bytes
    assert bench.traffic_for(1, W.scaled(dlrm, 26, 1), 100.0, str(path)) == 120.0  # the captured case itself
    assert bench.traffic_for(1, W.kg(), 200.0, str(path)) is None              # another workload
    assert bench.traffic_for(1, W.scaled(dlrm, 1, 2), 200.0, str(path)) is None  # another batch size
    assert bench.traffic_for(2, dlrm, 200.0, str(path)) is None                # no figure for the kernel
    path.write_text(json.dumps({"dlrm": {"1": dict(rec, source_sha="0" * 16)}}))
    assert bench.traffic_for(1, dlrm, 200.0, str(path)) is None                # kernel source changed since


def test_traffic_record_from_an_ncu_csv(tmp_path):
    """--traffic-record: per-launch DRAM bytes of each kernel class from ncu's
    CSV (units converted, launches averaged), beside the algorithmic bytes of
    the same launches' batch."""
    import argparse
    import json

    import workloads as W

    cfg = W.scaled(W.tiny(), 50, 4)
    hdr = ["ID", "Process ID", "Process Name", "Host Name", "Kernel Name", "Context", "Stream", "Block Size",
           "Grid Size", "Device", "CC", "Section Name", "Metric Name", "Metric Unit", "Metric Value"]

    def row(i, name, metric, unit, v):
        return [str(i), "1", "python", "h", name, "1", "7", "(256, 1, 1)", "(1, 1, 1)", "0", "10.3", "Command line",
                metric, unit, v]

    rows = [hdr,
            row(0, "void (anonymous namespace)::k_get<4, 1, 1>(IndexArgs)", "dram__bytes_read.sum", "Mbyte", "2.5"),
            row(0, "void (anonymous namespace)::k_get<4, 1, 1>(IndexArgs)", "dram__bytes_write.sum", "Kbyte", "500"),
            row(0, "void (anonymous namespace)::k_get<4, 1, 1>(IndexArgs)", "gpu__time_duration.sum", "usecond", "9"),
            row(1, "(anonymous namespace)::k_sort_scatter(const unsigned int *)", "dram__bytes_read.sum", "byte",
                "1,000"),
            row(1, "(anonymous namespace)::k_sort_scatter(const unsigned int *)", "dram__bytes_write.sum", "byte",
                "0"),
            row(2, "(anonymous namespace)::k_sort_scatter(const unsigned int *)", "dram__bytes_read.sum", "byte",
                "3,000"),
            row(2, "(anonymous namespace)::k_sort_scatter(const unsigned int *)", "dram__bytes_write.sum", "byte",
                "0")]
    csv_path = tmp_path / "launches.csv"
    csv_path.write_text("\n".join(",".join('"%s"' % c for c in r) for r in rows) + "\n")
    args = argparse.Namespace(pool=2, steps=1, warmup=3, scale=50)
    out_path = tmp_path / "traffic.json"
    out = bench.record_traffic(args, cfg, str(csv_path), str(out_path))
    assert out["1"]["bytes_per_launch"] == 3.0e6 and out["1"]["launches"] == 1
    assert out["3"]["bytes_per_launch"] == 2000.0 and out["3"]["launches"] == 2
    s = bench.batch_stats(cfg.batch_keys(1), cfg.dim)  # the timed step replays batch (3 + 0) % 2
    assert out["1"]["algorithmic_bytes_per_launch"] == bench.kernel_bytes(s, 1, 2)
    assert json.loads(out_path.read_text())[cfg.name]["3"]["source_sha"] == bench.source_sha(3)


def test_traffic_record_of_get_put_batches_uses_their_gets(tmp_path):
    """For the YCSB-shaped batches the Get reads only the batch's Get keys: the
    record's algorithmic bytes are those of ycsb_stats (what the bench's own
    roofline uses), not of every key of the batch."""
    import argparse

    import workloads as W

    cfg = W.scaled(W.ycsb(), 50_000, 64)  # 1,000 records, batches of 16,384 operations
    hdr = ["ID", "Process ID", "Process Name", "Host Name", "Kernel Name", "Context", "Stream", "Block Size",
           "Grid Size", "Device", "CC", "Section Name", "Metric Name", "Metric Unit", "Metric Value"]
    name = "void (anonymous namespace)::k_get<4, 2, 1>(IndexArgs)"
    rows = [hdr] + [[ "0", "1", "python", "h", name, "1", "7", "(256, 1, 1)", "(1, 1, 1)", "0", "10.3",
                      "Command line", m, "byte", "100"] for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")]
    csv_path = tmp_path / "launches.csv"
    csv_path.write_text("\n".join(",".join('"%s"' % c for c in r) for r in rows) + "\n")
    args = argparse.Namespace(pool=2, steps=1, warmup=3, scale=50_000)
    out = bench.record_traffic(args, cfg, str(csv_path), str(tmp_path / "traffic.json"))
    read, write, _ = cfg.ops(1)  # the timed step replays batch (3 + 0) % 2
    want = bench.kernel_bytes(bench.ycsb_stats(read, write, cfg.dim), 1, 1)
    assert out["1"]["algorithmic_bytes_per_launch"] == want
    assert want < bench.kernel_bytes(bench.batch_stats(cfg.batch_keys(1), cfg.dim), 1, 1)

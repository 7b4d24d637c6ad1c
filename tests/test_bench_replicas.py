"""bench.py's multi-GPU arithmetic on CPU: N replicas (one process each, gloo)
report the whole job's rate over the slowest rank's time, every rank agrees on
it, and the reference arm runs on rank 0 alone."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank), MLKV_BENCH_BACKEND="gloo")
    sys.path.insert(0, ROOT)
    import bench

    dist, r, local, w = bench.dist_setup(world)
    elapsed = 10.0 + 5.0 * r  # rank 1 is the slow one
    worst, value = bench.job_throughput(dist, torch, elapsed, 1_000, device="cpu")
    bench.barrier(dist, torch, sync_cuda=False)
    q.put((r, w, worst, value))
    dist.destroy_process_group()


def test_two_replicas_report_the_job_rate_over_the_slowest_rank():
    import torch.multiprocessing as mp

    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for r, w, worst, value in got:
        assert w == 2
        assert worst == 15.0                          # max over ranks, on every rank
        assert value == pytest.approx(2_000 / 0.015)  # both ranks' units over the slowest time


def _run_reference(rank, world):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    return subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny", "--steps", "2",
                           "--warmup", "3"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


def test_reference_arm_runs_on_rank_zero_only():
    r1 = _run_reference(1, 2)
    assert r1.returncode == 0 and r1.stdout.strip() == ""
    r0 = _run_reference(0, 2)
    assert r0.returncode == 0
    line = json.loads(r0.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["e2e"]["h2d_bytes_per_step"] == 0

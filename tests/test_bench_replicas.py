"""bench.py's multi-GPU path on CPU: N replicas (one process each, gloo)
report the whole job's rate over the slowest rank's time, every rank agrees on
it, `--gpus N` starts its own N ranks, and the reference arm prints from rank 0
alone."""
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


def test_gpus_flag_starts_its_own_ranks():
    """`bench.py --gpus 2` with no launcher environment starts two ranks itself;
    on the reference arm (no GPU work) both join one gloo group and rank 0 alone
    prints the line, with n_gpus = the group's size."""
    env = {k: v for k, v in os.environ.items()
           if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT")}
    r = subprocess.run([sys.executable, "bench.py", "--gpus", "2", "--impl", "reference", "--config", "tiny",
                        "--steps", "2", "--warmup", "3"], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout  # rank 0 only
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["n_gpus"] == 2 and line["config"]["parallelism"] == "replicas2"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["cpu_baseline"]["cpu_model"]


def test_rank_count_must_match_the_flag(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.setenv("WORLD_SIZE", "1")
    with pytest.raises(SystemExit):
        bench.dist_setup(2)

"""Benchmark of the batched embedding Get + gradient apply through the store.

One step = Get(keys) into a device buffer, then apply_grad(keys, grads) (one
Adagrad step per distinct key on its summed gradient), on the DLRM-shaped
store: 26 tables x 4,000,000 rows x dim 128 fp32 (rows + Adagrad state resident
in HBM, about 107 GB), 65,536 samples x 26 Zipf(1.2) lookups per step
(1,703,936 lookups).  Inputs are seeded and synthetic, generated before timing
and resident in HBM; each step's gradients (872 MB) and Get output (872 MB)
exceed the 129 MB L2, so no flush is needed between steps.

Prints one JSON line.  `value` is lookups (rows) per second of the whole job;
`e2e` is the same metric through the host-buffer C-ABI calls with the copies
inside the timed region; `roofline` is the dominant kernel's algorithmic bytes
per launch over its CUDA-event duration against the measured HBM copy peak;
`cpu_baseline` is the oracle (single thread, host cores) on a bounded sample.

With the default DLRM workload at N=1 the same process then measures the
knowledge-graph, GNN and tiered workloads and the YCSB-shaped Get/Put batches
(Zipf and uniform keys) one after another (each store closed before the next
opens) and reports them under `per_config`, each with its own metric, roofline,
clocks and oracle baseline.

`--gpus N` without a launcher's environment starts N replica ranks itself
(torch.distributed.run on this host, one process per GPU).

--impl reference times the oracle itself on the host, as the reference arm.
"""
import argparse
import ctypes
import gc
import hashlib
import json
import os
import platform
import socket
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "embedding rows/s (Get + grad-apply) and achieved HBM GB/s vs ~8 TB/s peak"
UNIT = "rows/s"
METRIC_YCSB = "key-value operations/s (YCSB-shaped batches of Gets and Puts)"
UNIT_YCSB = "ops/s"
NOMINAL_HBM_GBS = 8000.0
SEQ_SEGMENT_MAX = 32
SMALL_RUN = 4  # runs of 2 .. SMALL_RUN lookups go to k_small (their positions in their record)
CHUNK = 64


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# --- clocks during the timed region ---------------------------------------------
class ClockSampler:
    """Samples SM clock and clock-event reasons with nvidia-smi (-lms) and, where
    the driver's NVML library loads, a fast NVML poll.  NVML samples carry their
    host time, so the summary can say how many fell inside the timed region."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.samples = []  # (host time or None, sm_mhz, max_mhz, reasons_mask, source)
        self._stop = threading.Event()
        self._smi = None
        self._thread = None
        self._nvml = None
        self._handle = None
        self._get_reasons = None
        self.nvml_status = "not loaded"
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            rc = nv.nvmlInit_v2()
            if rc != 0:
                self.nvml_status = f"nvmlInit_v2 returned {rc}"
            else:
                h = ctypes.c_void_p()
                rc = nv.nvmlDeviceGetHandleByIndex_v2(gpu_index, ctypes.byref(h))
                fn = None
                for name in ("nvmlDeviceGetCurrentClocksEventReasons", "nvmlDeviceGetCurrentClocksThrottleReasons"):
                    try:
                        fn = getattr(nv, name)
                        break
                    except AttributeError:
                        continue
                if rc != 0:
                    self.nvml_status = f"nvmlDeviceGetHandleByIndex_v2 returned {rc}"
                elif fn is None:
                    self.nvml_status = "no clock-event-reasons entry point"
                else:
                    self._nvml, self._handle, self._get_reasons = nv, h, fn
                    self.nvml_status = "ok"
        except OSError as e:
            self.nvml_status = f"libnvidia-ml.so.1: {e}"

    def _poll(self):
        nv, h, reasons = self._nvml, self._handle, self._get_reasons
        clk, mx, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        while not self._stop.is_set():
            t = time.perf_counter()
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and \
                    nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0 and \
                    reasons(h, ctypes.byref(rs)) == 0:
                self.samples.append((t, clk.value, mx.value, rs.value, "nvml"))
            time.sleep(0.001)

    def start(self):
        try:
            # nvidia-smi's samples go to a temporary file, read back in stop()
            fd, self._smi_path = tempfile.mkstemp(prefix="mlkv_clocks_", suffix=".csv")
            os.close(fd)
            self._smi = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}",
                 "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self._smi_path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self._smi = None
        if self._nvml is not None:
            self._thread = threading.Thread(target=self._poll, daemon=True)
            self._thread.start()

    def stop(self):
        self._stop.set()
        if self._thread:
            self._thread.join()
        if self._smi:
            self._smi.terminate()
            self._smi.wait()
            try:
                for ln in open(self._smi_path):
                    f = [x.strip() for x in ln.split(",")]
                    if len(f) >= 5 and f[1].isdigit():
                        mask = int(f[4], 16) if f[4].startswith("0x") else 0
                        self.samples.append((None, int(f[1]), int(f[2]), mask, "nvidia-smi"))
            except OSError:
                pass
            try:
                os.remove(self._smi_path)
            except OSError:
                pass

    def summary(self, timed=None, window=None):
        """Median SM clock, max clock and the union of reasons over every sample
        of the window; `timed` = (t0, t1) host times of the timed region, to
        count the NVML samples inside it."""
        out = {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": len(self.samples),
               "nvml": self.nvml_status}
        if window:
            out["window"] = window
        if timed is not None:
            out["samples_in_timed_region"] = sum(1 for s in self.samples
                                                 if s[0] is not None and timed[0] <= s[0] <= timed[1])
        if not self.samples:
            return out
        mask = 0
        for s in self.samples:
            mask |= s[3]
        out.update(sm_mhz=statistics.median(s[1] for s in self.samples),
                   sm_max_mhz=max(s[2] for s in self.samples),
                   reasons=[v for k, v in sorted(self.REASONS.items()) if mask & k])
        return out


def sync_ok(store, what: str):
    """Waits for the store; a device status set by its kernels raises with the
    library's text of it."""
    rc = store.sync()
    if rc:
        raise RuntimeError(f"{what}: status {rc}: {store.lib.mlkv_last_error(store.h).decode()}")


def cpu_description() -> dict:
    """Model and count of the host's cores (lscpu, else /proc/cpuinfo)."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.lower().startswith("model name:"):
                model = ln.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if not model:
        try:
            for ln in open("/proc/cpuinfo"):
                if ln.lower().startswith("model name"):
                    model = ln.split(":", 1)[1].strip()
                    break
        except OSError:
            pass
    return {"cpu_model": model or platform.processor() or platform.machine(), "host_cores": os.cpu_count(),
            "machine": platform.machine()}


# --- workload statistics (algorithmic bytes) ----------------------------------------
def batch_stats(keys: np.ndarray, d: int) -> dict:
    """Exact per-kernel algorithmic bytes of one step on this batch."""
    _, counts = np.unique(keys, return_counts=True)
    B, U = len(keys), len(counts)
    long_ = counts > SEQ_SEGMENT_MAX
    Bl, Ul = int(counts[long_].sum()), int(long_.sum())
    Bs, Us = B - Bl, U - Ul
    U1 = int((counts == 1).sum())  # runs of one lookup (k_single)
    small = (counts >= 2) & (counts <= SMALL_RUN)
    Usm, Bsm = int(small.sum()), int(counts[small].sum())  # runs of 2 .. SMALL_RUN lookups (k_small)
    Bm, Um = Bs - U1 - Bsm, Us - U1 - Usm                  # the other short runs (k_short)
    items = int(np.ceil(counts[long_] / CHUNK).sum())
    row = 4 * d
    return {
        "B": B, "U": U, "Bs": Bs, "Us": Us, "Bl": Bl, "Ul": Ul, "items": items, "U1": U1, "Um": Um,
        "Usm": Usm, "Bsm": Bsm,
        # Get: keys + output per lookup; index sector + row per distinct key
        "get_gather": B * (8 + row) + U * (32 + row),
        # runs of SMALL_RUN + 1 .. 32 lookups: gradient rows + sorted position per
        # lookup; row and state read and written once plus the run's 16-byte record
        "reduce_short": Bm * (row + 4) + Um * (4 * row + 16),
        # runs of 2 .. SMALL_RUN lookups: gradient rows; row and state read and
        # written once, the 20-byte record with the run's positions
        "reduce_small": Bsm * row + Usm * (4 * row + 20),
        # runs of one lookup: the gradient row, row and state read and written
        # once, the 8-byte record
        "reduce_single": U1 * (row + 4 * row + 8),
        # long runs: gradient rows + sorted positions, chunk sums written
        "reduce_long": Bl * (row + 4) + items * row,
        # chunk sums read, row and state read and written once per long run
        "long_combine": items * row + Ul * 4 * row,
        # whole step, what the method must move: keys twice, output + grads per
        # lookup; index sector + Get row read + row/state RMW per distinct key
        "step": B * (16 + 2 * row) + U * (32 + 5 * row),
    }


def ycsb_stats(read: np.ndarray, write: np.ndarray, d: int) -> dict:
    """Algorithmic bytes of one Get + Put batch."""
    R, W = len(read), len(write)
    Ur, Uw = len(np.unique(read)), len(np.unique(write))
    row = 4 * d
    return {
        "B": R + W, "U": Ur + Uw,
        "get_gather": R * (8 + row) + Ur * (32 + row),     # keys + output; index sector + row per key
        "probe": W * 12 + Uw * 32,                         # the Put's keys and rows; index sector per key
        "put_scatter": W * (8 + row + 4) + Uw * row,       # value + row id + slot per write; row per key
        "step": R * (8 + row) + Ur * (32 + row) + W * (8 + row) + Uw * (32 + row),
    }


def kernel_bytes(stats: dict, kid: int, sort_passes: int) -> float:
    if "put_scatter" in stats:  # a key-value batch
        return {1: stats["get_gather"], 2: stats["probe"], 9: stats["put_scatter"]}[kid]
    if kid == 1:
        return stats["get_gather"]
    if kid == 4:
        return stats["reduce_short"]
    if kid == 10:
        return stats["reduce_single"]
    if kid == 11:
        return stats["reduce_small"]
    if kid == 5:
        return stats["reduce_long"]
    if kid == 7:
        return stats["long_combine"]
    if kid == 3:
        return stats["B"] * 16.0  # per pass: (row id, position) read and written
    if kid == 2:
        return stats["B"] * 12.0 + stats["U"] * 32.0
    if kid == 6:  # each sorted row id read twice and each position once; the run records written
        return stats["B"] * 12.0 + stats["U1"] * 8.0 + stats["Usm"] * 20.0 + stats["Um"] * 16.0
    return 0.0


KERNEL_NAMES = {1: "k_get (probe + row gather)", 2: "k_probe", 3: "k_sort_scatter",
                4: "k_short (run sum + Adagrad)", 5: "k_long_sum (chunk sums of long runs)",
                6: "k_heads (runs found in the sorted ids)", 7: "k_long_combine (chunk sums + Adagrad)",
                8: "k_tier_fetch (host <-> HBM row swap)", 9: "k_put_scatter (Put: last occurrence writes)",
                10: "k_single (runs of one lookup + Adagrad)", 11: "k_small (runs of 2-4 lookups + Adagrad)"}
KERNEL_SOURCES = {1: "mlkv_index.cu", 2: "mlkv_index.cu", 3: "mlkv_sort.cu", 4: "mlkv_apply.cu",
                  5: "mlkv_apply.cu", 6: "mlkv_apply.cu", 7: "mlkv_apply.cu", 8: "mlkv_tier.cu",
                  9: "mlkv_index.cu", 10: "mlkv_apply.cu", 11: "mlkv_apply.cu"}


# ncu kernel names (demangled, without the namespace) -> kernel class
KERNEL_PATTERNS = [("k_get_bulk<", 1), ("k_get<", 1), ("k_probe<", 2), ("k_sort_scatter", 3), ("k_short<", 4),
                   ("k_long_sum<", 5), ("k_heads", 6), ("k_long_combine<", 7), ("k_tier_fetch", 8),
                   ("k_put_scatter", 9), ("k_single<", 10), ("k_small<", 11)]
TRAFFIC_PATH = os.path.join(ROOT, "profiles", "traffic.json")


def kernel_id_of(name: str):
    for pat, kid in KERNEL_PATTERNS:
        if pat in name:
            return kid
    return None


def source_sha(kid: int) -> str:
    src = os.path.join(ROOT, "paper_2504_01506_gb300", "csrc", KERNEL_SOURCES[kid])
    return hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]


def traffic_for(kid: int, cfg, alg_bytes: float, path=None):
    """DRAM bytes (read + written) of one launch of kernel class `kid` in this
    workload, from the committed ncu record: the record must have been taken on
    the same workload and batch size (over the full table, or one `scale` times
    smaller, which keeps every input and output larger than L2) and on the
    kernel's current source (hash match).  The captured bytes are scaled to
    this launch by the algorithmic bytes (this launch's over the captured
    launches').  None when there is no such record."""
    try:
        with open(path or TRAFFIC_PATH) as f:
            rec = json.load(f).get(cfg.name, {}).get(str(kid))
    except (OSError, ValueError):
        return None
    if not rec or rec.get("batch_lookups") != cfg.batch or rec.get("source_sha") != source_sha(kid):
        return None
    a = rec.get("algorithmic_bytes_per_launch")
    return rec["bytes_per_launch"] * alg_bytes / a if a else None


def record_traffic(args, cfg, csv_path: str, path=None) -> dict:
    """Reads an ncu CSV (--metrics dram__bytes_read.sum,dram__bytes_write.sum
    --csv, launches of the timed steps of this same command line) and writes
    the per-launch DRAM bytes of each kernel class it holds, beside the
    algorithmic bytes of the same launches, into the traffic record of this
    workload.  No GPU work."""
    import csv

    unit = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9}
    per_launch = {}  # ncu launch ID -> [kernel name, bytes]
    with open(csv_path, newline="") as f:
        rows = [r for r in csv.reader(f) if len(r) > 10]
    hdr = rows[0]
    col = {h: i for i, h in enumerate(hdr)}
    for r in rows[1:]:
        if r[col["Metric Name"]] not in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            continue
        v = float(r[col["Metric Value"]].replace(",", "")) * unit[r[col["Metric Unit"]]]
        e = per_launch.setdefault(r[col["ID"]], [r[col["Kernel Name"]], 0.0])
        e[1] += v
    by_kid = {}
    for name, b in per_launch.values():
        kid = kernel_id_of(name)
        if kid is not None:
            by_kid.setdefault(kid, ([], name))[0].append(b)
    pool = max(1, min(args.pool, args.steps + args.warmup))
    steps_idx = [(args.warmup + i) % pool for i in range(args.steps)]
    if isinstance(cfg, W.YcsbConfig):  # a batch of Gets, then Puts (the bytes measure() uses)
        stats = {j: ycsb_stats(*cfg.ops(j)[:2], cfg.dim) for j in set(steps_idx)}
    else:
        stats = {j: batch_stats(cfg.batch_keys(j), cfg.dim) for j in set(steps_idx)}
    passes = -(-int(cfg.n_keys).bit_length() // 9)
    out = {}
    for kid, (bs, name) in sorted(by_kid.items()):
        alg = float(np.mean([kernel_bytes(stats[j], kid, passes) for j in steps_idx]))
        short = name.split("(")[0].replace("void ", "").replace("unnamed>::", "").replace("(anonymous namespace)::", "")
        out[str(kid)] = {"kernel": short.strip(),
                         "rows": cfg.n_keys, "scale": args.scale, "batch_lookups": cfg.batch,
                         "launches": len(bs), "bytes_per_launch": float(np.mean(bs)),
                         "algorithmic_bytes_per_launch": alg, "source": KERNEL_SOURCES[kid],
                         "source_sha": source_sha(kid)}
    path = path or TRAFFIC_PATH
    try:
        with open(path) as f:
            allrec = json.load(f)
    except (OSError, ValueError):
        allrec = {}
    allrec[cfg.name] = out
    with open(path, "w") as f:
        json.dump(allrec, f, indent=1, sort_keys=True)
        f.write("\n")
    return out


# --- distributed plumbing (replicas) --------------------------------------------------
def dist_setup(n_gpus: int):
    """This process's rank in a launched job (RANK / LOCAL_RANK / WORLD_SIZE from
    the launcher); a job of more than one rank joins a process group."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != n_gpus:
        raise SystemExit(f"--gpus {n_gpus} but the launcher started {world} rank(s)")
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if os.environ.get("MLKV_BENCH_BACKEND", "nccl") == "nccl" else "gloo"
        dist.init_process_group(backend=backend)
        return dist, rank, local, world
    return None, 0, 0, 1


def _free_port() -> int:
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def launch_replicas(n: int, argv) -> int:
    """`--gpus N` started without a launcher: re-runs this script as N ranks on
    this host (torch.distributed.run, rendezvous on 127.0.0.1), one per GPU, and
    returns the job's exit status.  Rank 0 prints the JSON line."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr=127.0.0.1", f"--master-port={_free_port()}", os.path.abspath(__file__), *argv]
    return subprocess.run(cmd, cwd=ROOT).returncode


def barrier(dist, torch, sync_cuda: bool = True):
    if dist is not None:
        dist.barrier()
    if sync_cuda:
        torch.cuda.synchronize()


def max_over_ranks(dist, torch, x: float, device: str = "cuda") -> float:
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(dist, torch, elapsed_ms: float, units_per_rank: float, device: str = "cuda"):
    """Whole-job rate of N replicas: all ranks' units over the slowest rank's time.
    Returns (slowest ms, units/s)."""
    world = dist.get_world_size() if dist is not None else 1
    worst = max_over_ranks(dist, torch, elapsed_ms, device)
    return worst, units_per_rank * world / (worst / 1e3)


# --- the oracle arms -------------------------------------------------------------------
def oracle_steps(cfg, steps: int, sample: int, warmup: int = 0):
    """Times the oracle (one host thread) on `steps` Get + apply steps, each on
    the first `sample` lookups of that step's batch.  Returns (lookups/s, seconds)."""
    import oracle

    ref = oracle.Table(cfg.dim, lr=cfg.lr, eps=cfg.eps, state_init=cfg.state_init, init_lo=cfg.init_lo,
                       init_hi=cfg.init_hi, seed=cfg.seed, precision=32)
    batches = [(cfg.batch_keys(s)[:sample], cfg.grads(s, sample)) for s in range(warmup + steps)]
    for k, g in batches[:warmup]:
        ref.get(k)
        ref.apply_grad(k, g)
    t0 = time.perf_counter()
    for k, g in batches[warmup:]:
        ref.get(k)
        ref.apply_grad(k, g)
    dt = time.perf_counter() - t0
    ref.close()
    return steps * sample / dt, dt


def oracle_ycsb_steps(cfg, steps: int, sample: int, warmup: int = 0):
    """Times the oracle (one host thread) on `steps` Get + Put batches, each on
    the first `sample` operations of that step's batch.  Returns (ops/s, seconds)."""
    import oracle

    ref = oracle.Table(cfg.dim, precision=32, seed=cfg.seed, init_lo=cfg.init_lo, init_hi=cfg.init_hi)
    batches = []
    for s in range(warmup + steps):
        r, w, v = cfg.ops(s)
        nr = int(round(sample * len(r) / cfg.batch))
        batches.append((r[:nr], w[:sample - nr], v[:sample - nr]))
    for r, w, v in batches[:warmup]:
        ref.get(r)
        ref.put(w, v)
    t0 = time.perf_counter()
    for r, w, v in batches[warmup:]:
        ref.get(r)
        ref.put(w, v)
    dt = time.perf_counter() - t0
    return steps * sample / dt, dt


def run_reference(args, cfg):
    """The reference arm: the oracle on one host thread, rank 0 only.  Under N
    ranks every rank joins a gloo group (no GPU work), so the line's n_gpus is
    the job's world size; the other ranks do nothing else."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but the launcher started {world} rank(s)")
    dist = None
    if world > 1:
        import datetime

        import torch.distributed as dist

        dist.init_process_group(backend="gloo", timeout=datetime.timedelta(minutes=30))
        world = dist.get_world_size()
    if rank == 0:
        sample = max(1, cfg.batch // 8)
        kv = isinstance(cfg, W.YcsbConfig)
        value, dt = (oracle_ycsb_steps if kv else oracle_steps)(cfg, args.steps, sample, args.warmup)
        line = {
            "impl": "reference", "metric": METRIC_YCSB if kv else METRIC, "value": value,
            "unit": UNIT_YCSB if kv else UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": dict(workload_config(cfg), parallelism=f"replicas{world}"),
            "cpu_baseline": dict({"value": value, "unit": UNIT_YCSB if kv else UNIT, "cores": 1, "kind": "oracle",
                                  "sample": f"first {sample} of {cfg.batch} operations of each step"},
                                 **cpu_description()),
            "e2e": {"value": value, "unit": UNIT_YCSB if kv else UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
        }
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def dma_peak(torch, dev) -> dict:
    """Pinned host <-> device copy bandwidth (1 GiB, best of 3), GB/s."""
    n = 1 << 28
    h = torch.empty(n, dtype=torch.float32).pin_memory()
    d = torch.empty(n, dtype=torch.float32, device=dev)
    out = {}
    for name, fn in (("h2d", lambda: d.copy_(h, non_blocking=True)), ("d2h", lambda: h.copy_(d, non_blocking=True))):
        best = 0.0
        for _ in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            best = max(best, 4 * n / (e0.elapsed_time(e1) / 1e3) / 1e9)
        out[name] = best
    return out


def workload_config(cfg) -> dict:
    where = (f"in host memory behind an HBM cache of {cfg.hbm_cache_rows:,} rows" if cfg.hbm_cache_rows
             else "in HBM")
    c = {"workload": f"{cfg.name}: {cfg.n_keys:,} rows x dim {cfg.dim} fp32 (+ Adagrad state) {where}, "
                     f"{cfg.batch:,} lookups/step",
         "rows": cfg.n_keys, "dim": cfg.dim, "batch_lookups": cfg.batch, "lr": cfg.lr,
         "l2": "inputs larger than L2 every step (gradients and Get output 4*dim B per lookup)"}
    if isinstance(cfg, W.configs.DlrmConfig):
        c.update({"tables": cfg.tables, "zipf_alpha": cfg.alpha})
    if isinstance(cfg, W.YcsbConfig):
        keys = f"Zipf({cfg.alpha})" if cfg.alpha else "uniform"
        c = {"workload": f"{cfg.name}: {cfg.n_keys:,} records of {cfg.dim} fp32 in HBM, batches of "
                         f"{cfg.batch:,} operations ({cfg.read_fraction:.0%} Get, the rest Put), {keys} keys",
             "records": cfg.n_keys, "dim": cfg.dim, "batch_ops": cfg.batch, "read_fraction": cfg.read_fraction,
             "keys": keys, "l2": "inputs larger than L2 every step (written values and Get output 1 KiB per op)"}
    return c


# --- our arm ----------------------------------------------------------------------------
CLOCK_WINDOW_S = 1.0  # clocks are sampled over the timed region and, after it, the same steps to this length


def measure(args, cfg, dist, rank, local, world, dev, headline: bool, steps: int) -> dict:
    """Opens the store of `cfg`, preloads it, times `steps` Get + apply steps (or
    Get + Put batches) and returns the measured fields; the store is closed on
    return.  `headline`: also the end-to-end host-buffer leg."""
    import torch

    from paper_2504_01506_gb300 import EmbeddingStore

    hbm_peak, peak_kind = peaks()
    t_begin = time.perf_counter()
    tiered = cfg.hbm_cache_rows > 0
    kv = isinstance(cfg, W.YcsbConfig)
    staleness = args.staleness if headline else 0
    store = EmbeddingStore(dim=cfg.dim, capacity=cfg.n_keys, max_batch=cfg.batch, lr=cfg.lr, eps=cfg.eps,
                           state_init=cfg.state_init, init_lo=cfg.init_lo, init_hi=cfg.init_hi,
                           seed=cfg.seed, hbm_cache_rows=cfg.hbm_cache_rows,
                           staleness_bound=staleness, device=dev)
    # stale-synchronous steps: each Get on one stream, each apply on another; the
    # table lets Get(t) run beside the last `staleness` applies before it
    s_get = torch.cuda.Stream(dev) if staleness else None
    s_apply = torch.cuda.Stream(dev) if staleness else None
    # preload every key of the table (untimed), in preload order
    chunk = cfg.batch
    for s0 in range(0, cfg.n_keys, chunk):
        store.insert(torch.from_numpy(cfg.preload_keys(s0, s0 + chunk)).to(dev))
    sync_ok(store, "preload failed")

    if tiered and args.tier_prefill:
        # fill the HBM cache with rows of random keys, each updated once (so the
        # cache starts full, as in a long run, and the timed steps evict)
        rng = np.random.default_rng(5)
        fill = rng.choice(cfg.n_keys, size=min(cfg.hbm_cache_rows, cfg.n_keys), replace=False).astype(np.int64)
        zeros = torch.zeros((cfg.batch, cfg.dim), dtype=torch.float32, device=dev)
        for s0 in range(0, len(fill), cfg.batch):
            k = torch.from_numpy(fill[s0:s0 + cfg.batch]).to(dev)  # tiered keys are 0..n_keys-1
            store.get(k)
            store.apply_grad(k, zeros[:k.numel()])
        sync_ok(store, "prefill failed")
        del zeros

    # The HBM store cycles a pool of batches.  The tiered store gets a fresh batch
    # every step (a cycled pool would end up resident in its cache): one per
    # kernel-class prepass step, warm-up step, timed step, and the last look-ahead.
    kinds = (1, 2, 9) if kv else (1, 2, 3, 4, 5, 6, 7, 10, 11) + ((8,) if tiered else ())
    base = len(kinds) if tiered else 0
    pool = base + args.warmup + steps + 1 if tiered else max(1, min(args.pool, steps + args.warmup))
    ngrad = max(1, min(args.pool, pool))
    out = torch.empty((cfg.batch, cfg.dim), dtype=torch.float32, device=dev)
    passes = -(-int(cfg.n_keys).bit_length() // 9)  # the sort's passes: digits of at most 9 bits
    if kv:  # batches of Gets, then Puts
        ops_d = []
        stats = []
        for s0 in range(pool):
            r, w, v = cfg.ops(s0)
            ops_d.append((torch.from_numpy(r).to(dev), torch.from_numpy(w).to(dev), torch.from_numpy(v).to(dev)))
            stats.append(ycsb_stats(r, w, cfg.dim))
        keys_h = None
    else:
        keys_h = [cfg.batch_keys(s0) for s0 in range(pool)]
        keys_d = [torch.from_numpy(k).to(dev) for k in keys_h]
        gen = torch.Generator(device=dev)
        grads_d = []
        for s0 in range(ngrad):
            gen.manual_seed(cfg.seed * 1000 + s0)
            grads_d.append(torch.randn((cfg.batch, cfg.dim), generator=gen, device=dev) * cfg.grad_sigma)
        stats = [batch_stats(k, cfg.dim) for k in keys_h]

    def step(i):
        j = i % pool
        if kv:
            r, w, v = ops_d[j]
            store.get(r, out=out[:r.numel()])
            store.put(w, v)
            return
        if staleness:
            with torch.cuda.stream(s_get):
                store.get(keys_d[j], out=out)
            with torch.cuda.stream(s_apply):
                store.apply_grad(keys_d[j], grads_d[i % ngrad])
            return
        store.get(keys_d[j], out=out)
        if tiered and args.lookahead:  # Lookahead(next keys) runs beside this step's apply
            store.lookahead(keys_d[(i + 1) % pool])
        store.apply_grad(keys_d[j], grads_d[i % ngrad])

    # pick the dominant kernel: one step per kernel class, timed with events
    kernel_ms = {}
    for idx, kid in enumerate(kinds):
        store.time_kernel(kid)
        step(idx if tiered else 0)
        ms, n = store.kernel_time()
        kernel_ms[kid] = ms
    store.time_kernel(0)
    dominant = max(kernel_ms, key=kernel_ms.get)
    for i in range(args.warmup):
        step(base + i)
    sync_ok(store, "device status")

    # An HBM-resident step is captured into a CUDA graph per batch (the Get and
    # the apply of that batch) and replayed: the calls' work is device-driven,
    # so a replay does all of it with one launch from the host.
    use_graphs = not tiered and args.graphs and not staleness  # stale-synchronous calls refuse capture
    graphs, launches_per_graph = [], 0
    if use_graphs:
        cap = torch.cuda.Stream(dev)
        l0 = store.launch_count()
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(cap):
            for j in range(pool):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=cap):
                    step(j)
                graphs.append(g)
        torch.cuda.synchronize(dev)
        launches_per_graph = (store.launch_count() - l0) // pool
        for i in range(args.warmup):
            graphs[(base + i) % pool].replay()
        sync_ok(store, "device status")

    def timed_step(i):
        if use_graphs:
            graphs[i % pool].replay()
        else:
            step(i)

    stream = torch.cuda.current_stream(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    if not use_graphs:
        store.time_kernel(dominant)
    launches0 = store.launch_count()
    tier0 = store.tier_stats()
    barrier(dist, torch)
    clocks.start()
    if args.profile:
        torch.cuda.profiler.start()
    t_timed0 = time.perf_counter()
    ev0.record(stream)
    for side in (s_get, s_apply):
        if side is not None:
            side.wait_stream(stream)
    for i in range(steps):
        timed_step(base + args.warmup + i)
    for side in (s_get, s_apply):
        if side is not None:
            stream.wait_stream(side)
    ev1.record(stream)
    barrier(dist, torch)
    t_timed1 = time.perf_counter()
    if args.profile:
        torch.cuda.profiler.stop()
    launches = launches_per_graph * steps if use_graphs else store.launch_count() - launches0
    tier1 = store.tier_stats()
    if not use_graphs:  # the dominant kernel's launches of the timed region
        dom_ms, dom_n = store.kernel_time()
        store.time_kernel(0)
    # a timed region shorter than the clock window: the sampler keeps running over
    # the same steps (untimed) right after it, so the record has enough samples
    n_extra = 0
    while time.perf_counter() - t_timed0 < CLOCK_WINDOW_S and n_extra < 100_000:
        for i in range(8):
            timed_step(base + args.warmup + (n_extra + i) % steps)
        n_extra += 8
        torch.cuda.synchronize(dev)
    clocks.stop()
    window = (f"the timed region ({steps} steps) and {n_extra} more of the same steps right after it "
              f"({time.perf_counter() - t_timed0:.2f} s)" if n_extra else f"the timed region ({steps} steps)")
    clock_summary = clocks.summary(timed=(t_timed0, t_timed1), window=window)
    sync_ok(store, "device status set during the timed region")
    elapsed_ms, value = job_throughput(dist, torch, ev0.elapsed_time(ev1), cfg.batch * steps)
    roof_region_ms = elapsed_ms
    if use_graphs:
        # event timings inside a graph are overwritten at every replay: the
        # dominant kernel is timed over the same steps run call by call
        store.time_kernel(dominant)
        r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        for i in range(steps):
            step(base + args.warmup + i)
        r1.record(stream)
        torch.cuda.synchronize(dev)
        roof_region_ms = r0.elapsed_time(r1)
        dom_ms, dom_n = store.kernel_time()
        store.time_kernel(0)
    sync_ok(store, "device status set during the roofline region")
    kernel_avg = None
    if args.kernel_times:
        # every kernel class event-timed over the same steps run call by call
        kernel_avg = {}
        for kid in kinds:
            store.time_kernel(kid)
            for i in range(steps):
                step(base + args.warmup + i)
            ms, n = store.kernel_time()
            kernel_avg[KERNEL_NAMES[kid]] = {"ms_per_step": ms / steps, "launches_per_step": n / steps}
        store.time_kernel(0)
        sync_ok(store, "device status")
    step_bytes = np.mean([st["step"] for st in stats])
    achieved_step = step_bytes * steps / (elapsed_ms / 1e3) / 1e9

    # roofline of the dominant kernel over the timed region
    avg_ms = dom_ms / max(dom_n, 1)
    tier = None
    if tiered:
        slot_bytes = 2 * ((cfg.dim + 7) // 8 * 8) * 4
        fetched, written = tier1[0] - tier0[0], tier1[1] - tier0[1]
        link_bytes = (fetched + written) * slot_bytes
        link_gbs = link_bytes / (elapsed_ms / 1e3) / 1e9
        peak = dma_peak(torch, dev)
        tier = {"host_rows": cfg.n_keys, "cache_rows": cfg.hbm_cache_rows, "rows_fetched_per_step": fetched / steps,
                "rows_written_back_per_step": written / steps,
                "sweep_lines_per_step": (tier1[2] - tier0[2]) / steps,
                "link_bytes_per_step": link_bytes / steps, "link_gbs_over_step": link_gbs,
                "dma_peak_gbs": peak, "lookahead": bool(args.lookahead), "prefilled": bool(args.tier_prefill)}
    if dominant == 8:
        # the swap kernel moves each fetched row in and each victim out over the
        # host link (its launches timed over the timed region)
        per_launch_bytes = link_bytes / max(dom_n, 1)
        achieved = per_launch_bytes / (avg_ms / 1e3) / 1e9
        roofline = {"bound": "host-link", "kernel": KERNEL_NAMES[8], "achieved": achieved, "peak": peak["h2d"],
                    "unit": "GB/s", "frac": achieved / peak["h2d"],
                    "peak_kind": "measured in this run (pinned cudaMemcpyAsync H2D, 1 GiB, sequential)",
                    "traffic": None, "bytes_per_launch": per_launch_bytes, "avg_launch_ms": avg_ms,
                    "launches": dom_n, "share_of_step": dom_ms / roof_region_ms if roof_region_ms else None}
    else:
        steps_idx = [(base + args.warmup + i) % pool for i in range(steps)]
        per_launch_bytes = np.mean([kernel_bytes(stats[j], dominant, passes) for j in steps_idx])
        achieved = per_launch_bytes / (avg_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "kernel": KERNEL_NAMES[dominant], "achieved": achieved, "peak": hbm_peak,
                    "unit": "GB/s", "frac": achieved / hbm_peak, "peak_kind": peak_kind,
                    "traffic": traffic_for(dominant, cfg, per_launch_bytes), "bytes_per_launch": per_launch_bytes,
                    "avg_launch_ms": avg_ms, "launches": dom_n,
                    "share_of_step": dom_ms / roof_region_ms if roof_region_ms else None,
                    "timed_over": "the timed steps run call by call right after the graph-replayed ones"
                    if use_graphs else "the timed region"}

    # end to end through the host-buffer calls (copies inside the timed region)
    e2e = None
    if headline and not args.no_e2e and kv:
        # keys and written values from pinned host memory, the Get's output back,
        # around the store's calls
        r, w, v = ops_d[0]
        hr, hw, hv = r.cpu().pin_memory(), w.cpu().pin_memory(), v.cpu().pin_memory()
        hout = torch.empty((r.numel(), cfg.dim), dtype=torch.float32).pin_memory()
        dr, dw, dv = torch.empty_like(r), torch.empty_like(w), torch.empty_like(v)
        e2e_steps = max(1, min(steps, 20))

        def kv_e2e():
            dr.copy_(hr, non_blocking=True)
            dw.copy_(hw, non_blocking=True)
            dv.copy_(hv, non_blocking=True)
            store.get(dr, out=out[:dr.numel()])
            store.put(dw, dv)
            hout.copy_(out[:dr.numel()], non_blocking=True)

        for _ in range(2):
            kv_e2e()
        barrier(dist, torch)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(e2e_steps):
            kv_e2e()
        e1.record(stream)
        barrier(dist, torch)
        e_ms = max_over_ranks(dist, torch, e0.elapsed_time(e1))
        sync_ok(store, "device status")
        h2d = (r.numel() + w.numel()) * 8 + v.numel() * 4
        d2h = r.numel() * cfg.dim * 4
        e2e = {"value": cfg.batch * e2e_steps * world / (e_ms / 1e3), "unit": UNIT_YCSB, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": e2e_steps,
               "link_gbs": (h2d + d2h) * e2e_steps / (e_ms / 1e3) / 1e9}
    if headline and not args.no_e2e and not tiered and not kv:
        e2e_pool = min(pool, 2)
        hk = [torch.from_numpy(keys_h[j]).pin_memory() for j in range(e2e_pool)]
        hg = [grads_d[j % ngrad].cpu().pin_memory() for j in range(e2e_pool)]
        hout = torch.empty((cfg.batch, cfg.dim), dtype=torch.float32).pin_memory()
        e2e_steps = max(1, min(steps, 20))
        for i in range(2):
            store.get_host(hk[i % e2e_pool], hout)
            store.apply_grad_host(hk[i % e2e_pool], hg[i % e2e_pool])
        barrier(dist, torch)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(e2e_steps):
            store.get_host(hk[i % e2e_pool], hout)
            store.apply_grad_host(hk[i % e2e_pool], hg[i % e2e_pool])
        e1.record(stream)
        barrier(dist, torch)
        e_ms = max_over_ranks(dist, torch, e0.elapsed_time(e1))
        sync_ok(store, "device status")
        h2d = cfg.batch * 8 * 2 + cfg.batch * cfg.dim * 4
        d2h = cfg.batch * cfg.dim * 4
        e2e = {"value": cfg.batch * e2e_steps * world / (e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": e2e_steps,
               "link_gbs": (h2d + d2h) * e2e_steps / (e_ms / 1e3) / 1e9}
    store.close()
    del graphs, out
    if not kv:
        del keys_d, grads_d
    else:
        del ops_d
    gc.collect()
    torch.cuda.empty_cache()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = max(1, cfg.batch // 8)
        csteps = max(1, args.cpu_steps)
        v, dt = (oracle_ycsb_steps if kv else oracle_steps)(cfg, csteps, sample)
        cpu = dict({"value": v, "unit": UNIT_YCSB if kv else UNIT, "cores": 1, "kind": "oracle",
                    "sample": f"{csteps} steps x first {sample} of {cfg.batch} "
                              f"{'operations (Get + Put)' if kv else 'lookups (Get + apply)'}, "
                              f"{dt:.1f} s on one host thread"}, **cpu_description())

    res = {
        "value": value, "ms_per_step": elapsed_ms / steps, "steps": steps,
        "config": dict(workload_config(cfg), parallelism=f"replicas{world}", distinct_batches=pool,
                       **({"staleness_bound": staleness} if staleness else {})),
        "achieved_gbs": achieved_step, "hbm_frac_measured": achieved_step / hbm_peak,
        "hbm_frac_nominal": achieved_step / NOMINAL_HBM_GBS,
        "distinct_per_step": float(np.mean([st["U"] for st in stats])),
        "distinct_rows_per_s": float(np.mean([st["U"] for st in stats])) * world * steps / (elapsed_ms / 1e3),
        "roofline": roofline, "kernel_ms_one_step": {KERNEL_NAMES[k]: v for k, v in kernel_ms.items()},
        **({"kernel_ms_avg": kernel_avg} if kernel_avg else {}),
        "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": launches, "clocks": clock_summary,
        "step_launch": (f"one CUDA graph replay per step (the Get and the {'Put' if kv else 'apply'} of the "
                        f"batch, captured)" if use_graphs else
                        "each call launched from the host" + (", Gets and applies on two streams"
                                                              if staleness else "")),
        "wall_s": time.perf_counter() - t_begin,
    }
    if tier is not None:
        res["tier"] = tier
    return res


def per_config_names(args, world) -> list:
    if args.per_config == "none" or world > 1:
        return []
    if args.per_config == "auto":
        if args.config != "dlrm" or args.scale != 1 or args.staleness:
            return []
        return ["kg", "gnn", "tiered", "ycsb", "ycsb-uniform"]
    return [c for c in args.per_config.split(",") if c]


def tier_scaled(cfg, args):
    """The tiered workload with its host tier scaled to the machine's host memory
    (and the HBM cache with it: the same cached fraction of the rows)."""
    full_rows, full_cache = cfg.n_keys, cfg.hbm_cache_rows
    cfg.n_keys = args.tier_rows
    cfg.hbm_cache_rows = args.tier_cache_rows or int(full_cache * args.tier_rows / full_rows)
    return cfg


def run_ours(args, cfg):
    import torch

    dist, rank, local, world = dist_setup(args.gpus)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    kv = isinstance(cfg, W.YcsbConfig)
    res = measure(args, cfg, dist, rank, local, world, dev, headline=True, steps=args.steps)
    extra = {}
    for name in per_config_names(args, world):
        c = W.ALL[name]()
        if name == "tiered":
            c = tier_scaled(c, args)
        # each workload's own step count (the timed region stays short), at most --steps
        r = measure(args, c, dist, rank, local, world, dev, headline=False, steps=min(args.steps, c.steps))
        r.pop("e2e", None)
        kvc = isinstance(c, W.YcsbConfig)
        r["metric"] = METRIC_YCSB if kvc else METRIC
        r["unit"] = UNIT_YCSB if kvc else UNIT
        extra[name] = r
    if rank == 0:
        line = {
            "metric": METRIC_YCSB if kv else METRIC, "value": res["value"], "unit": UNIT_YCSB if kv else UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": res["ms_per_step"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        }
        line.update({k: v for k, v in res.items() if k not in ("value", "ms_per_step", "steps")})
        if extra:
            line["per_config"] = extra
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="dlrm", choices=sorted(W.ALL))
    ap.add_argument("--pool", type=int, default=8, help="distinct pre-generated batches, cycled")
    ap.add_argument("--cpu-steps", type=int, default=6)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile", action="store_true",
                    help="bracket the timed region with cudaProfilerStart/Stop (ncu --profile-from-start off)")
    ap.add_argument("--tier-rows", type=int, default=96_000_000,
                    help="tiered config: rows of the host tier (1 KiB each with state)")
    ap.add_argument("--tier-cache-rows", type=int, default=0,
                    help="tiered config: rows cached in HBM (default: the workload's 120 GB cache over "
                         "400M rows, scaled with --tier-rows)")
    ap.add_argument("--no-tier-prefill", dest="tier_prefill", action="store_false",
                    help="tiered config: start with an empty HBM cache")
    ap.add_argument("--no-graphs", dest="graphs", action="store_false",
                    help="HBM-resident configs: launch each call from the host instead of replaying a CUDA graph")
    ap.add_argument("--no-lookahead", dest="lookahead", action="store_false",
                    help="tiered config: no look-ahead; each Get fetches its own missing rows")
    ap.add_argument("--scale", type=int, default=1,
                    help="divide the table's rows by this (same batch); for small profiling cases")
    ap.add_argument("--kernel-times", action="store_true",
                    help="also event-time every kernel class over the timed steps (run call by call)")
    ap.add_argument("--per-config", default="auto",
                    help="workloads measured after the headline one in the same process, comma-separated "
                         "(auto: kg,gnn,tiered,ycsb,ycsb-uniform after the default DLRM workload at N=1; "
                         "none: no others)")
    ap.add_argument("--traffic-record", metavar="CSV",
                    help="write the DRAM bytes per launch in this ncu CSV (dram__bytes_read.sum and "
                         "dram__bytes_write.sum of this command line's timed steps) into profiles/traffic.json "
                         "and exit (no GPU work)")
    ap.add_argument("--staleness", type=int, default=0,
                    help="HBM-resident training configs: open the table with this staleness bound (>= 1; "
                         "9223372036854775807 = asynchronous) and run Gets and applies on two streams")
    args = ap.parse_args()
    if args.staleness and (args.config in ("tiered", "ycsb", "ycsb-uniform") or args.staleness < 0):
        ap.error("--staleness takes a bound >= 1 and an HBM-resident training config")
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.gpus < 1:
        ap.error("--gpus must be >= 1")
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # no launcher: start the N replica ranks here
        return launch_replicas(args.gpus, sys.argv[1:])
    cfg = W.ALL[args.config]()
    if args.config == "tiered":
        # the host tier must fit the machine's host memory
        cfg = tier_scaled(cfg, args)
    if args.scale > 1:
        cfg = W.scaled(cfg, args.scale, 1)
    if args.traffic_record:
        print(json.dumps(record_traffic(args, cfg, args.traffic_record)))
        return 0
    if args.impl == "reference":
        return run_reference(args, cfg)
    return run_ours(args, cfg)


if __name__ == "__main__":
    sys.exit(main())

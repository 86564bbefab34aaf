"""Benchmark of the memory-planning path on GB300: one JSON line on stdout.

A step is one pass of the whole path -- live-bytes profile, greedy_by_size
plan (with its peak) and pairwise validation -- over the batched workload of
4096 random traces (512 tensors over T = 1024 steps each, seeds 0..4095; rank
r of a multi-GPU run takes seeds r*4096 .. r*4096+4095: weak scaling, no
collective on the data path).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--policy first|best]
    python bench.py --impl reference ...   # the CPU oracle as the reference arm
    python bench.py --all-configs          # every workload, one line each (not the bench line)

Timing: W untimed warm-up steps; then K steps, each preceded by an L2 flush
(256 MiB device write, outside the timed events) and timed with CUDA events
on the launching stream; barrier + synchronize on both sides of the K-step
region; the max over ranks is reported.  Per-kernel events give the dominant
kernel's achieved bandwidth for the roofline object.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "greedy-by-size tensors planned/s and validated pairs/s on 1 GB300 (% HBM roofline)"
UNIT = "tensors/s"
WORKLOAD = dict(n_traces=4096, n=512, T=1024, p=0.5, lo_e=6, hi_e=20)
WORKLOAD_NAME = "batched-random-4096x512x1024-seeds0-4095"
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 256 << 20

# Algorithmic bytes per unit (what each kernel must move at minimum).
# profile : read alloc/free/size 16 B per tensor and trace_ptr/steps/profile_ptr 20 B
#           per trace; write 8 B per step, peak_lb 8 B and status 4 B per trace.
# plan    : read 16 B per tensor and 12 B per trace; write offsets 8 B per tensor,
#           plan_peak 8 B and status 4 B per trace.
# validate: read alloc/free/size/offset 24 B per tensor and 12 B per trace; write
#           verdict 4 B, conflict 8 B and status 4 B per trace.
# fused   : read 16 B per tensor and 20 B per trace; write the profile 8 B per step,
#           offsets 8 B per tensor, and peak_lb, plan_peak, verdict, conflict and
#           status (32 B) per trace.
# bump    : read 16 B per tensor and 12 B per trace; write offsets 8 B per tensor,
#           plan_peak 8 B and status 4 B per trace.
KERNELS = ("live_profile", "plan_greedy_by_size", "validate_plan")
FUSED = "plan_and_validate"
# mp_plan_and_validate launches the planner kernel twice: once with 32-bit byte
# arithmetic over every trace, then once with 64-bit bytes for the traces whose
# sizes sum to 2^32 or more (a grid that walks the statuses and skips the rest).
LAUNCHES_PER_FUSED_CALL = 2


def algorithmic_bytes(kernel: str, n_tensors: int, n_traces: int, n_steps: int) -> int:
    if kernel == "live_profile":
        return 16 * n_tensors + 8 * n_steps + (20 + 12) * n_traces
    if kernel == "plan_greedy_by_size":
        return 24 * n_tensors + (12 + 12) * n_traces
    if kernel == "validate_plan":
        return 24 * n_tensors + (12 + 16) * n_traces
    if kernel == FUSED:
        return 24 * n_tensors + 8 * n_steps + (20 + 32) * n_traces
    if kernel in ("plan_bump", "plan_greedy_by_breadth"):
        return 24 * n_tensors + (12 + 12) * n_traces
    raise KeyError(kernel)


# ----------------------------------------------------------------- distributed helpers

def dist_env():
    """(rank, world, local_rank) from the torchrun environment (1 process if absent)."""
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def resolve_launch(gpus: int, env=None) -> str:
    """How this process should honour --gpus N: "run" (the ranks already match:
    one process for N = 1, or N torchrun ranks), "spawn" (N > 1 asked for
    without torchrun: re-launch this command under torch.distributed.run with N
    ranks) or "mismatch" (torchrun started a different number of ranks than
    --gpus asks for: refuse rather than report the wrong n_gpus)."""
    env = os.environ if env is None else env
    if gpus < 1:
        return "mismatch"
    if "WORLD_SIZE" not in env:
        return "run" if gpus == 1 else "spawn"
    return "run" if int(env["WORLD_SIZE"]) == gpus else "mismatch"


def spawn_ranks(gpus: int, argv) -> int:
    """Re-runs this script under torch.distributed.run with one rank per GPU
    (rendezvous on 127.0.0.1) and returns its exit status."""
    import socket

    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={gpus}",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__), *argv]
    return subprocess.call(cmd)


def shard_seed0(rank: int, n_traces: int = WORKLOAD["n_traces"]) -> int:
    """First seed of this rank's batch (weak scaling: every rank plans its own batch)."""
    return rank * n_traces


def max_over_ranks(value: float, dist=None) -> float:
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return value
    import torch

    backend = dist.get_backend()
    dev = torch.device("cuda", torch.cuda.current_device()) if backend == "nccl" else torch.device("cpu")
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, dist=None) -> float:
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return value
    import torch

    backend = dist.get_backend()
    dev = torch.device("cuda", torch.cuda.current_device()) if backend == "nccl" else torch.device("cpu")
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ----------------------------------------------------------------- measurement helpers

def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# The sources the fused planner kernel is built from (its traffic in
# profiles/ncu_traffic.json holds only while these are unchanged).
PLANNER_SOURCES = ("plan.cu", "common.cuh", "launch.h")


def kernel_source_digest() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2203_00448_gb300", "csrc")
    for fn in PLANNER_SOURCES:
        h.update(open(os.path.join(csrc, fn), "rb").read())
    return h.hexdigest()


def ncu_record(kernel: str, n_tensors: int, field: str = "dram_bytes"):
    """A per-launch counter (DRAM bytes, warp instructions) from the committed
    ncu capture, scaled to this launch's tensor count; None if absent or if the
    kernels changed since."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except (OSError, ValueError):
        return None
    if d.get("source_sha256") != kernel_source_digest():
        return None
    k = d.get("kernels", {}).get(kernel)
    if not k or field not in k:
        return None
    return k[field] * n_tensors / k["n_tensors"]


# Each SM has four schedulers that issue one warp instruction per cycle each.
ISSUE_PER_SM_PER_CLK = 4


def issue_roofline(warp_inst: float, seconds: float, n_sms: int, sm_mhz: float):
    """Second roofline for the integer planner, which is issue-bound rather than
    HBM-bound: warp instructions per second against n_sms * 4 * clock."""
    if warp_inst is None or not sm_mhz:
        return None
    peak = n_sms * ISSUE_PER_SM_PER_CLK * sm_mhz * 1e6
    achieved = warp_inst / seconds
    return {"bound": "issue", "achieved": achieved, "peak": peak, "unit": "warp-inst/s", "frac": achieved / peak,
            "warp_inst_per_launch": warp_inst,
            "peak_source": f"{n_sms} SMs x {ISSUE_PER_SM_PER_CLK} warp-inst/clk x {sm_mhz:.0f} MHz (median SM clock "
                           f"sampled during the timed steps)",
            "inst_source": "smsp__inst_executed.sum of the committed ncu capture, scaled by tensors"}


def gpu_id(dev) -> str:
    """The device's UUID ("GPU-..."), as NVML and nvidia-smi --id accept it."""
    import torch

    uuid = getattr(torch.cuda.get_device_properties(dev), "uuid", None)
    if uuid is not None:
        u = str(uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    return str(dev.index or 0)


class ClockSampler:
    """SM clock and throttle-reason sampling during the timed region.

    Reads NVML (read-only queries) from a background thread every millisecond;
    falls back to `nvidia-smi -lms 100` if NVML cannot be loaded.
    """

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown"}
    SMI_QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_uuid: str):
        self.uuid = gpu_uuid
        self.samples = []  # (sm_mhz, max_mhz, reasons bitmask)
        self.proc = None
        self.thread = None
        self.stop = False
        self.nvml = self._open_nvml()

    def _open_nvml(self):
        import ctypes

        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return None
            h = ctypes.c_void_p()
            if lib.nvmlDeviceGetHandleByUUID(self.uuid.encode(), ctypes.byref(h)) != 0:
                return None
            reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
            return lib, h, reasons
        except (OSError, AttributeError):
            return None

    def _poll(self):
        import ctypes

        lib, h, reasons = self.nvml
        clk, mx, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        while not self.stop:
            if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and \
                    lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0 and reasons(h, ctypes.byref(rs)) == 0:
                self.samples.append((clk.value, mx.value, rs.value))
            time.sleep(0.001)

    def sample_now(self):
        """One reading from the calling thread (between timed steps)."""
        if self.nvml is None:
            return
        import ctypes

        lib, h, reasons = self.nvml
        clk, mx, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and \
                lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0 and reasons(h, ctypes.byref(rs)) == 0:
            self.samples.append((clk.value, mx.value, rs.value))

    def __enter__(self):
        import threading

        if self.nvml is not None:
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
        else:
            try:
                self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.uuid}", f"--query-gpu={self.SMI_QUERY}",
                                              "--format=csv,noheader,nounits", "-lms", "100"],
                                             stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            except OSError:
                self.proc = None
        return self

    def __exit__(self, *exc):
        if self.thread is not None:
            self.stop = True
            self.thread.join(timeout=2)
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
            bits = {"hw_slowdown": 0x8, "hw_thermal_slowdown": 0x40, "sw_thermal_slowdown": 0x20, "sw_power_cap": 0x4}
            for r in (out or "").strip().splitlines():
                c = [x.strip() for x in r.split(",")]
                if len(c) >= 9 and c[1].isdigit() and c[2].isdigit():
                    mask = sum(bits[names[k]] for k in range(4) if c[5 + k] == "Active")
                    self.samples.append((int(c[1]), int(c[2]), mask))

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm = [x[0] for x in self.samples]
        reasons = sorted({name for x in self.samples for bit, name in self.REASONS.items() if x[2] & bit})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(x[1] for x in self.samples), "reasons": reasons,
                "samples": len(self.samples), "source": "nvml" if self.nvml is not None else "nvidia-smi"}


# ----------------------------------------------------------------- CPU oracle baseline

def oracle_baseline(ts, n_sample_traces: int):
    """The oracle as it stands, single-threaded on the host: profile + plan +
    validate over the first `n_sample_traces` traces of the workload."""
    import oracle

    sub = ts.select(range(min(n_sample_traces, ts.n_traces)))
    t0 = time.perf_counter()
    oracle.live_profile(sub)
    off, _, _ = oracle.plan_greedy_by_size(sub, oracle.FIT_FIRST)
    oracle.validate_plan(sub, off)
    dt = time.perf_counter() - t0
    return sub.n_tensors / dt, dt, sub


def _oracle_path_seconds(ts):
    """Profile + plan (first fit) + validate of a TraceSet with the oracle; the seconds taken."""
    import oracle

    t0 = time.perf_counter()
    oracle.live_profile(ts)
    off, _, _ = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    oracle.validate_plan(ts, off)
    return time.perf_counter() - t0


def oracle_pool(cores: int):
    """A spawn-started process pool for the all-cores oracle leg (spawned, so it
    is safe whenever it is created; created before the first GPU call)."""
    import multiprocessing as mproc

    import tracegen

    pool = mproc.get_context("spawn").Pool(cores)
    pool.map(_oracle_path_seconds, [tracegen.random_small(1, 2, 4, 8)] * cores)  # workers up, oracle loaded
    return pool


def oracle_all_cores(ts, pool, cores: int):
    """The oracle as it stands over the whole batch, its traces split into
    `cores` interleaved parts run by `cores` processes at once; wall seconds."""
    n_parts = min(cores, ts.n_traces)
    parts = [ts.select(range(c, ts.n_traces, n_parts)) for c in range(n_parts)]
    t0 = time.perf_counter()
    pool.map(_oracle_path_seconds, parts)
    return time.perf_counter() - t0, n_parts


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import tracegen

    w = WORKLOAD
    ts = tracegen.random_batch(0, w["n_traces"], w["n"], w["T"], w["p"], w["lo_e"], w["hi_e"], name=WORKLOAD_NAME)
    sample = 512
    for _ in range(args.warmup):
        oracle_baseline(ts, sample)
    times, n = [], 0
    for _ in range(args.steps):
        _, dt, sub = oracle_baseline(ts, sample)
        times.append(dt)
        n = sub.n_tensors
    total = sum(times)
    value = n * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic", "config": {"workload": WORKLOAD_NAME, "policy": "first", "n_traces_per_step": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"first {sample} of the 4096 traces per step (profile + plan + validate)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ----------------------------------------------------------------- GPU arm

def run_gpu(args):
    rank, world, local = dist_env()
    cores = os.cpu_count() or 1
    pool = oracle_pool(cores) if (rank == 0 and args.oracle_traces > 0 and world == 1) else None
    import torch

    dist = None
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    import paper_2203_00448_gb300 as mp
    import tracegen
    from paper_2203_00448_gb300 import build

    build.build()
    w = WORKLOAD
    ts = tracegen.random_batch(shard_seed0(rank, args.traces), args.traces, w["n"], w["T"], w["p"], w["lo_e"],
                               w["hi_e"], name=WORKLOAD_NAME if args.traces == w["n_traces"] else
                               f"batched-random-{args.traces}x512x1024")
    dev = torch.device("cuda", torch.cuda.current_device())
    db = mp.DeviceBatch.from_host(ts, dev)
    buf = mp.PathBuffers(db)
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step(ev):
        ev[0].record(stream)
        mp.plan_and_validate(db, args.policy, buf, stream=stream)
        ev[1].record(stream)

    def step_separate(ev):
        ev[0].record(stream)
        mp.live_profile(db, buf.profile, buf.peak_lb, buf.status[0], stream=stream)
        ev[1].record(stream)
        mp.plan_greedy_by_size(db, args.policy, buf.offsets, buf.plan_peak, buf.status[1], workspace=buf.plan_ws,
                               stream=stream)
        ev[2].record(stream)
        mp.validate_plan(db, buf.offsets, buf.verdict, buf.conflict, buf.status[2], workspace=buf.validate_ws,
                         stream=stream)
        ev[3].record(stream)

    mk = lambda k: [torch.cuda.Event(enable_timing=True) for _ in range(k)]
    for _ in range(args.warmup):
        flush.zero_()
        step(mk(2))
        if not args.no_breakdown:
            flush.zero_()
            step_separate(mk(4))
    torch.cuda.synchronize()
    step(mk(2))
    torch.cuda.synchronize()
    if not bool((buf.status[0] == 0).all()) or not bool((buf.verdict == 1).all()):
        print(json.dumps({"error": "path reported a failed trace or an invalid plan", "rank": rank}))
        return 1

    events = [mk(2) for _ in range(args.steps)]
    sampler = ClockSampler(gpu_id(dev))
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with sampler:
        t0 = time.perf_counter()
        for k in range(args.steps):
            flush.zero_()
            step(events[k])
            sampler.sample_now()  # between steps: the host is not inside any timed pair of events
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    if dist is not None:
        dist.barrier()
    step_times = [ev[0].elapsed_time(ev[1]) for ev in events]
    step_ms = statistics.median(step_times)
    step_ms_mean = statistics.fmean(step_times)
    step_ms_max = max_over_ranks(step_ms, dist)
    wall_max = max_over_ranks(wall, dist)
    total_tensors = sum_over_ranks(float(ts.n_tensors), dist)
    total_pairs = sum_over_ranks(float(ts.pairs()), dist)

    # The same step as three separate kernels (profile, plan, validate), for the breakdown.
    per_kernel = [float("nan")] * 3
    if not args.no_breakdown:
        sep_events = [mk(4) for _ in range(max(3, args.steps // 2))]
        for ev in sep_events:
            flush.zero_()
            step_separate(ev)
        torch.cuda.synchronize()
        per_kernel = [sum(ev[j].elapsed_time(ev[j + 1]) for ev in sep_events) / len(sep_events) for j in range(3)]

    # Rows beyond the hot path, timed the same way on the same batch:
    # bump_allocation (the baseline strategy of Sec. 2.3).
    next_rows = None
    if not args.no_breakdown:
        bump_off = torch.empty_like(buf.offsets)
        bump_pk = torch.empty_like(buf.plan_peak)
        bump_st = torch.empty_like(buf.status[0])
        for _ in range(args.warmup):
            mp.plan_bump(db, bump_off, bump_pk, bump_st, stream=stream)
        bump_events = [mk(2) for _ in range(max(3, args.steps // 2))]
        for ev in bump_events:
            flush.zero_()
            ev[0].record(stream)
            mp.plan_bump(db, bump_off, bump_pk, bump_st, stream=stream)
            ev[1].record(stream)
        torch.cuda.synchronize()
        if not bool((bump_st == 0).all()):
            print(json.dumps({"error": "plan_bump reported a failed trace", "rank": rank}))
            return 1
        bump_ms = sum(ev[0].elapsed_time(ev[1]) for ev in bump_events) / len(bump_events)
        next_rows = {"plan_bump": {"ms": bump_ms}}
        # greedy by breadth on the same batch, and its plan peaks against greedy_by_size's
        br_off = torch.empty_like(buf.offsets)
        br_pk = torch.empty_like(buf.plan_peak)
        br_st = torch.empty_like(buf.status[0])
        bws = mp.Workspace(dev)
        mp.plan_greedy_by_breadth(db, args.policy, br_off, br_pk, br_st, workspace=bws, stream=stream)
        br_events = [mk(2) for _ in range(3)]
        for ev in br_events:
            flush.zero_()
            ev[0].record(stream)
            mp.plan_greedy_by_breadth(db, args.policy, br_off, br_pk, br_st, workspace=bws, stream=stream)
            ev[1].record(stream)
        torch.cuda.synchronize()
        if not bool((br_st == 0).all()):
            print(json.dumps({"error": "plan_greedy_by_breadth reported a failed trace", "rank": rank}))
            return 1
        pk_ratio = br_pk.double() / buf.plan_peak.double()
        next_rows["plan_greedy_by_breadth"] = {
            "ms": sum(ev[0].elapsed_time(ev[1]) for ev in br_events) / len(br_events),
            "peak_over_greedy_by_size": {"mean": float(pk_ratio.mean()), "min": float(pk_ratio.min()),
                                         "max": float(pk_ratio.max())}}
        # The exact optimum on small traces (the generator of the bench
        # workload, 9 tensors over 6 steps, so that lifetimes overlap) and the
        # gap of the greedy plan to it.
        small = tracegen.random_batch(1 << 20, 4096, 9, 6, name="random-4096x9x6")
        sdb = mp.DeviceBatch.from_host(small, dev)
        ows = mp.Workspace(dev)
        o_off, o_pk, o_st = mp.plan_optimal(sdb, workspace=ows, stream=stream)
        g_off, g_pk, g_st = mp.plan_greedy_by_size(sdb, args.policy, stream=stream)
        torch.cuda.synchronize()
        opt_events = [mk(2) for _ in range(3)]
        for ev in opt_events:
            ev[0].record(stream)
            mp.plan_optimal(sdb, o_off, o_pk, o_st, workspace=ows, stream=stream)
            ev[1].record(stream)
        torch.cuda.synchronize()
        if not (bool((o_st == 0).all()) and bool((g_st == 0).all())):
            print(json.dumps({"error": "plan_optimal reported a failed trace", "rank": rank}))
            return 1
        ratio = g_pk.double() / o_pk.double()
        next_rows["plan_optimal"] = {
            "ms": sum(ev[0].elapsed_time(ev[1]) for ev in opt_events) / len(opt_events),
            "workload": small.name, "orders_per_trace": 362880,
            "greedy_over_optimum": {"policy": args.policy, "mean": float(ratio.mean()), "max": float(ratio.max()),
                                    "share_optimal": float((ratio == 1).double().mean())}}

    # End to end through the host-buffer API: pinned H2D of the inputs, the
    # path, and D2H of every result, each step.
    e2e = None
    if not args.no_e2e:
        hp = mp.HostPath(ts, dev, args.policy, stream=stream, chunks=args.e2e_chunks)
        hp.stage(ts)
        for _ in range(max(1, args.warmup)):
            hp.run()
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        e2e_steps = max(3, args.steps // 2)
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            hp.run()
        e2e_s = max_over_ranks((time.perf_counter() - t0) / e2e_steps, dist)
        e2e = {"value": total_tensors / e2e_s, "unit": UNIT, "h2d_bytes_per_step": hp.h2d_bytes,
               "d2h_bytes_per_step": hp.d2h_bytes, "ms_per_step": 1e3 * e2e_s,
               "call": f"mp_plan_and_validate_host, {hp.chunks} chunks, pinned host buffers, host wall clock"}

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0
    peak, peak_kind = measured_peaks()
    n_steps = ts.n_steps
    kern = None if args.no_breakdown else {}
    for j, name in enumerate(KERNELS if not args.no_breakdown else ()):
        nbytes = algorithmic_bytes(name, ts.n_tensors, ts.n_traces, n_steps)
        gbs = nbytes / (per_kernel[j] * 1e-3) / 1e9
        kern[name] = {"ms": per_kernel[j], "algorithmic_bytes": nbytes, "achieved_gbs": gbs, "frac": gbs / peak}
    if next_rows is not None:
        for name, row in next_rows.items():
            if name not in ("plan_bump", "plan_greedy_by_breadth"):
                continue  # the exhaustive search is bound by its n! placements, not by memory
            nbytes = algorithmic_bytes(name, ts.n_tensors, ts.n_traces, n_steps)
            gbs = nbytes / (row["ms"] * 1e-3) / 1e9
            row.update({"algorithmic_bytes": nbytes, "achieved_gbs": gbs, "frac": gbs / peak})
    fused_bytes = algorithmic_bytes(FUSED, ts.n_tensors, ts.n_traces, n_steps)
    fused_gbs = fused_bytes / (step_ms * 1e-3) / 1e9
    traffic = ncu_record(FUSED, ts.n_tensors)
    roof = {"bound": "hbm",
            "kernel": "k_plan, fused profile + plan + validate (one mp_plan_and_validate call: the 32-bit launch "
                      "and the 64-bit launch, which returns at once on this workload)",
            "achieved": fused_gbs, "peak": peak, "unit": "GB/s", "frac": fused_gbs / peak,
            "peak_source": f"{peak_kind} ({'MEASURED_PEAKS.json hbm_gbs' if peak_kind == 'measured' else 'profiling-recipe fallback'})",
            "algorithmic_bytes_per_launch": fused_bytes, "traffic": traffic}
    if args.oracle_traces > 0:
        ob_value, ob_dt, ob_sub = oracle_baseline(ts, args.oracle_traces)
        single = {"value": ob_value, "unit": UNIT, "cores": 1, "kind": "oracle",
                  "sample": f"first {ob_sub.n_traces} of {ts.n_traces} traces, profile + plan + validate, "
                            f"{ob_dt:.2f} s single-threaded"}
        if pool is not None:
            wall_all, n_parts = oracle_all_cores(ob_sub, pool, cores)
            cpu_baseline = {"value": ob_sub.n_tensors / wall_all, "unit": UNIT, "cores": n_parts, "kind": "oracle",
                            "sample": f"first {ob_sub.n_traces} of {ts.n_traces} traces, profile + plan + validate, "
                                      f"split over {n_parts} processes on {cores} host cores, {wall_all:.2f} s wall",
                            "single_core": single}
        else:
            cpu_baseline = single
    else:
        cpu_baseline = None
    if pool is not None:
        pool.close()
        pool.join()
    clocks = sampler.summary()
    issue = issue_roofline(ncu_record(FUSED, ts.n_tensors, "warp_inst"), step_ms * 1e-3,
                           torch.cuda.get_device_properties(dev).multi_processor_count,
                           clocks["sm_mhz"] or clocks["sm_max_mhz"])
    line = {
        "metric": METRIC, "value": total_tensors / (step_ms_max * 1e-3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms_max, "ms_per_step_mean": step_ms_mean,
        "ms_per_step_min": min(step_times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": ts.name if world == 1 else WORKLOAD_NAME, "n_traces": ts.n_traces * world,
                   "tensors_per_trace": w["n"],
                   "steps_per_trace": w["T"], "policy": args.policy,
                   "l2": "flushed before every timed step (256 MiB device write outside the timed events)",
                   "timing": f"median over ranks' median of {args.steps} event-timed steps",
                   "parallelism": f"dp{world} (traces sharded by rank, no collective)"},
        "validated_pairs_per_s": total_pairs / (step_ms_max * 1e-3),
        "wall_ms_per_step_incl_flush": 1e3 * wall_max / args.steps,
        "gpu_launches": args.steps * LAUNCHES_PER_FUSED_CALL,
        "separate_kernels_ms_per_step": None if args.no_breakdown else sum(per_kernel),
        "separate_kernels": kern,
        "next_rows": next_rows,
        "roofline": roof,
        "issue_roofline": issue,
        "cpu_baseline": cpu_baseline,
        "e2e": e2e,
        "clocks": clocks,
    }
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_all_configs(args):
    """Every workload of tracegen.CONFIG_NAMES through one mp_plan_and_validate
    call, timed like the bench step, next to the oracle on 1 host core and on
    all host cores (traces split over processes).  One JSON line per workload;
    these are parity workloads with their own shapes, not the bench line."""
    import torch

    import paper_2203_00448_gb300 as mp
    import tracegen
    from paper_2203_00448_gb300 import build

    cores = os.cpu_count() or 1
    pool = oracle_pool(cores)  # before the first GPU call
    build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    peak, peak_kind = measured_peaks()
    stream = torch.cuda.current_stream()
    for k in sorted(tracegen.CONFIG_NAMES):
        if args.config is not None and k != args.config:
            continue
        ts = tracegen.config(k)
        db = mp.DeviceBatch.from_host(ts, dev)
        buf = mp.PathBuffers(db)
        for _ in range(args.warmup):
            mp.plan_and_validate(db, args.policy, buf, stream=stream)
        times = []
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            mp.plan_and_validate(db, args.policy, buf, stream=stream)
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
        ok = bool((buf.status[0] == 0).all()) and bool((buf.verdict == 1).all())
        ms = statistics.median(times)
        nbytes = algorithmic_bytes(FUSED, ts.n_tensors, ts.n_traces, ts.n_steps)
        one_core = all_cores = n_chunks = None
        if args.oracle_traces > 0:  # 0: a profiling run, no oracle legs
            one_core = _oracle_path_seconds(ts)
            all_cores, n_chunks = oracle_all_cores(ts, pool, cores)
        gbs = nbytes / (ms * 1e-3) / 1e9
        print(json.dumps({
            "workload": tracegen.CONFIG_NAMES[k], "policy": args.policy, "ok": ok, "n_traces": ts.n_traces,
            "n_tensors": ts.n_tensors, "ms_per_call": ms, "tensors_per_s": ts.n_tensors / (ms * 1e-3),
            "validated_pairs_per_s": ts.pairs() / (ms * 1e-3),
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                         "peak_source": peak_kind, "algorithmic_bytes": nbytes},
            "oracle_1core_s": one_core, "oracle_all_cores_s": all_cores, "oracle_cores": n_chunks,
            "timing": f"median of {args.steps} calls after {args.warmup} warm-up, L2 flushed before each"}),
            flush=True)
    pool.close()
    pool.join()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--policy", choices=("first", "best"), default="first")
    ap.add_argument("--oracle-traces", type=int, default=4096,
                    help="traces of the workload the CPU-baseline leg runs through the oracle")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-chunks", type=int, default=4,
                    help="runs of traces the end-to-end call pipelines its copies over")
    ap.add_argument("--no-breakdown", action="store_true",
                    help="skip the three-kernel breakdown (profiling runs that should launch the fused kernel only)")
    ap.add_argument("--traces", type=int, default=WORKLOAD["n_traces"],
                    help="traces per rank (the reported workload is the default 4096; other values are for profiling)")
    ap.add_argument("--all-configs", action="store_true",
                    help="time every workload (one JSON line each) beside the oracle on 1 and on all host cores "
                         "(--oracle-traces 0 leaves the oracle out)")
    ap.add_argument("--config", type=int, default=None,
                    help="with --all-configs: that workload only (tracegen.CONFIG_NAMES)")
    args = ap.parse_args(argv)
    if args.all_configs:
        return run_all_configs(args)
    if args.impl == "reference":
        return run_reference(args)
    how = resolve_launch(args.gpus)
    if how == "spawn":
        return spawn_ranks(args.gpus, sys.argv[1:] if argv is None else list(argv))
    if how == "mismatch":
        print(json.dumps({"error": f"--gpus {args.gpus} but WORLD_SIZE={os.environ.get('WORLD_SIZE')}: launch one "
                                   f"rank per GPU (torchrun --nproc-per-node {args.gpus}) or drop torchrun"}))
        return 2
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())

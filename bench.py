"""Benchmark of the RPD commit step on GB300.

Default workload (N=1): the LLaDA-8B-shaped first step - batch 1, a 256-position canvas
all masked, K=4 window layers, d=4096, V=126464 (1024 projected rows), tau 0.9, budget
1.0 - with synthetic seeded inputs (the calibrated hidden-state recipe of ``workloads``).
One "step" is one rpd_step call: gather + RMSNorm prologue, tcgen05 head statistics,
split merge, scoring/scan/commit.  The step clears committed positions of its mask, so
every timed step reads its own copy of the input mask, written before the timed region:
each step sees the same workload and the timed region holds nothing but the steps.

Metric: commit steps/s (and rows/s).  Under torchrun each rank runs its own canvas
(weak scaling, no collective on the data path; a barrier and a max-reduce of the timer
only).  The default line also carries the decode trajectory at the same head shape (every
layer projected, and the projection chosen per step on the device) and the CPU oracle's
rate on a bounded sample of the workload, single-threaded and with every host core.
``--impl reference`` times whole steps of the CPU oracle on the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "RPD commit steps/s & rows/s at LLaDA-8B head shape; % of bf16 TC/HBM roofline"
UNIT = "commit-steps/s"

# DRAM bytes (read + write) per head-statistics launch from ncu captures, keyed by workload
# and by a hash of the kernel's sources at capture time; any source change makes it null.
HEAD_SOURCES = ("paper_2609_36452_gb300/csrc/k_head_stats.cu", "paper_2609_36452_gb300/csrc/ptx.cuh",
                "paper_2609_36452_gb300/csrc/rpd_internal.h", "paper_2609_36452_gb300/csrc/head_plan.h")
HEAD_TRAFFIC = {
    ("llada_first_step", "38d1ebfe76e73880"): 1.0519e9,
    ("llada_tail_70_masked", "38d1ebfe76e73880"): 1.0551e9,
    ("llada_tail_5_masked", "38d1ebfe76e73880"): 1.0404e9,
    ("dream_mid_decode", "38d1ebfe76e73880"): 1.1035e9,
    ("batched_serving", "38d1ebfe76e73880"): 8.8575e9,
}

# Nominal dense rates of GB300 (context only; the fractions use the measured peaks).
NOMINAL_BF16_TFLOPS = 2250.0
NOMINAL_HBM_GBS = 7900.0


def head_source_hash() -> str:
    import hashlib
    h = hashlib.sha256()
    for rel in HEAD_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm_gbs=p["hbm_gbs"], bf16_tflops=p["bf16_tflops"],
                    bf16_tflops_sustained=p.get("bf16_tflops_sustained", p["bf16_tflops"]),
                    source="measured")
    return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0, source="fallback")


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class ClockSampler:
    """nvidia-smi samples of SM clock, power and throttle reasons, every 100 ms."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (FileNotFoundError, OSError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for _, ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def make_workload(rank: int, masked: int = 0, window: int = 0):
    """The LLaDA first-step canvas; ``masked`` > 0 keeps only the last ``masked`` positions
    masked (the few-rows, head-streaming regime at the end of a decode trajectory);
    ``window`` > 0 projects that many final layers instead of 4 (16 is the paper's LLaDA
    window, App. A.6)."""
    import workloads as WL
    W, g = WL.make_head(WL.LLADA_V, WL.LLADA_D, seed=2)
    case = WL.llada_first_step(seed=2 + 97 * rank, W=W, g=g, K=window or 4)
    if window:
        case["name"] = f"llada_first_step_window{window}"
    if masked:
        m = torch.zeros(case["N"], dtype=torch.uint8)
        m[case["N"] - masked:] = 1
        case["mask"] = m
        case["name"] = f"llada_tail_{masked}_masked"
    return case


def rows_of(case):
    return case["K"] * int(case["mask"].sum())


def work_per_step(case):
    """Algorithmic work of one step: FLOPs of the head contraction and the bytes of the
    head (read once) plus the masked hidden rows."""
    R = rows_of(case)
    d, V = case["d"], case["V"]
    flops = 2.0 * R * d * V
    bytes_ = 2.0 * V * d + 2.0 * R * d
    return R, flops, bytes_


def blas_threads() -> int:
    """Threads the oracle's BLAS runs with (threadpoolctl where installed, else the thread
    variables BLAS libraries read, else every host core)."""
    try:
        from threadpoolctl import threadpool_info
        blas = [i for i in threadpool_info() if i.get("user_api") == "blas"]
        if blas:
            return int(blas[0].get("num_threads", 1))
    except Exception:
        pass
    for var in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    return os.cpu_count() or 1


def oracle_step_seconds(case, positions: int) -> float:
    """Wall time of one oracle step (as it stands) over the first ``positions`` canvas
    positions of the workload (``positions`` = N: the whole step)."""
    from oracle import rpd_oracle as O
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)  # noqa: E731
    hb = bits(case["hidden"][:, :positions])
    mask = case["mask"][:positions].numpy().astype(np.uint8)
    Wb, gb = bits(case["W"]), bits(case["g"])
    t0 = time.perf_counter()
    O.rpd_step(hb, mask, gb, Wb, case["eps"], case["tau"], case["budget"], case["rule"])
    return time.perf_counter() - t0


def single_thread_oracle_rate(positions: int, timeout_s: float = 600.0):
    """Rows/s of the oracle with one BLAS thread, on the first ``positions`` positions of the
    LLaDA first step, timed in a child process started with the BLAS thread variables set to 1
    (a BLAS library reads them when it loads).  Returns (rows/s, seconds) or None."""
    code = ("import json, sys; sys.path.insert(0, %r); import torch; "
            "torch.set_num_threads(max(1, __import__('os').cpu_count() or 1)); "
            "import bench; c = bench.make_workload(0); "
            "dt = bench.oracle_step_seconds(c, %d); "
            "print(json.dumps({'rows': c['K'] * %d, 'seconds': dt, 'threads': bench.blas_threads()}))"
            % (ROOT, positions, positions))
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1", BLIS_NUM_THREADS="1",
               VECLIB_MAXIMUM_THREADS="1")
    try:
        r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                           timeout=timeout_s)
        out = json.loads(r.stdout.strip().splitlines()[-1])
    except Exception:
        return None
    return out["rows"] / out["seconds"], out["seconds"], out["threads"]


def run_reference(args):
    """The CPU oracle, as it stands, on the LLaDA first step: every warm-up and timed step is
    one whole oracle step (256 masked positions, 1024 rows, full V and d; full logits in fp64)
    with the BLAS threads of the host."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    case = make_workload(0)
    R, flops, bytes_ = work_per_step(case)
    N = case["N"]
    for _ in range(args.warmup):
        oracle_step_seconds(case, N)
    times = [oracle_step_seconds(case, N) for _ in range(args.steps)]
    total = sum(times)
    steps_s = args.steps / total
    threads = blas_threads()
    out = {
        "impl": "reference", "metric": METRIC, "value": steps_s, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": config_dict(case, R),
        "rows_per_s": steps_s * R,
        "cpu_baseline": {"value": steps_s, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{args.warmup} warm-up + {args.steps} timed whole oracle steps "
                                   f"({R} rows each, full V and d, logits in fp64) with {threads} "
                                   f"BLAS threads on {os.cpu_count()} host cores; median step "
                                   f"{1e3 * statistics.median(times):.0f} ms"},
        "e2e": {"value": steps_s, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out))


def launches_per_step(case, args) -> int:
    """Kernels one rpd_step / rpd_step_batched call launches: the compaction; per projection
    pass gather/norm, the head kernel and the merge; the band selection before a second (lazy)
    pass; and score/commit, which the last merge performs itself for a single canvas of at
    most 2048 positions."""
    B = case.get("B", 1)
    K, N = case["K"], case["N"]
    second_pass = args.projection == "lazy" or (args.projection == "auto" and K > 1 and K * B * N > 256)
    fused_score = B == 1 and N <= 2048
    return 1 + 3 * (2 if second_pass else 1) + (1 if second_pass else 0) + (0 if fused_score else 1)


def config_dict(case, R):
    B = case.get("B", 1)
    rule = case["rule"]
    return {"workload": case["name"], "batch": B, "N": case["N"], "K": case["K"],
            "d": case["d"], "V": case["V"], "rows": R, "tau": case["tau"], "budget": case["budget"],
            "rule": f"{rule} (Table 4)" if "block" not in rule else f"{rule} (Table 4, RPD-block 32)",
            "signal_kappa": case.get("kappa"),
            "projection": "lazy" if "lazy_rows" in case else "all window layers",
            "rows_projected": case.get("lazy_rows", R),
            "head_tiling": case.get("tiling", "auto (per pass, on the device)"),
            "head_layout": case.get("head_layout", "tiled (context copy of W in contiguous 128 x 64 blocks)"),
            "l2": f"inputs larger than L2: the {2 * case['V'] * case['d'] / 1e9:.2f} GB head is streamed every step"}


def load_workload(args, rank):
    """The benchmarked workload for this rank (each rank draws its own canvases)."""
    import workloads as WL
    if args.workload == "llada_first_step":
        case = make_workload(rank, args.masked, args.window)
    elif args.workload == "dream_mid_decode":
        case = WL.dream_mid_decode(seed=3 + 97 * rank)
    elif args.workload == "batched_serving":
        case = WL.batched_serving(seed=5 + 97 * rank)
    else:
        raise ValueError(args.workload)
    if args.block:
        case["rule"] = case["rule"] + "_block"
        case["name"] = case["name"] + "_rpd_block"
    return case


def masked_rows(case):
    """Projected rows of one step: K x masked positions (RPD-block: the active blocks only)."""
    import workloads as WL  # noqa: F401
    masks = case["mask"].reshape(-1, case["N"])
    rows = 0
    for m in masks:
        idx = torch.nonzero(m).flatten()
        if "block" in case["rule"] and len(idx):
            lo = (int(idx[0]) // 32) * 32
            idx = idx[(idx >= lo) & (idx < lo + 32)]
        rows += case["K"] * len(idx)
    return rows


def aggregate_timing(ms_total_local: float, steps: int, world: int, reduce_max):
    """Whole-job timing: the slowest rank's time for ``steps`` steps on every rank, and the
    aggregate throughput (every rank ran its own canvases)."""
    ms_total = float(reduce_max(ms_total_local))
    return ms_total, ms_total / steps, world * steps / (ms_total / 1e3)


def run_rpd(args):
    rank, world, local = dist_env()
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    import paper_2609_36452_gb300 as rpd

    case = load_workload(args, rank)
    K, N, d, V = case["K"], case["N"], case["d"], case["V"]
    B = case.get("B", 1)
    R = masked_rows(case)
    flops = 2.0 * R * d * V
    bytes_ = 2.0 * V * d + 2.0 * R * d
    W = case["W"].to(dev)
    g = case["g"].to(dev)
    hidden = case["hidden"].to(dev).contiguous()
    mask0 = case["mask"].to(dev)
    # The step clears committed positions of its mask in place.  Every step of a timed pass
    # gets its own copy of the input mask, written before the pass starts, so the timed
    # region holds the steps alone (no reset copies between them).
    n_masks = max(args.steps, args.warmup)
    masks = mask0.unsqueeze(0).repeat(n_masks, *([1] * mask0.dim())).contiguous()
    commit = torch.zeros(B, N, dtype=torch.uint8, device=dev)
    token = torch.full((B, N), -1, dtype=torch.int32, device=dev)
    stats = torch.zeros(B, rpd.STATS_WORDS, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    ctx = rpd.Rpd(d, V, K, case["eps"])
    ctx.set_stream(stream)
    ctx.set_head_layout(args.head_layout)
    ctx.set_head(W, g)
    ctx.set_profile(case["rule"])
    ctx.reserve(B, N)
    ctx.set_projection(args.projection)
    ctx.set_head_tiling(args.tiling)
    if args.tiling != "auto":
        case["name"] = case["name"] + "_" + args.tiling
        case["tiling"] = args.tiling
    if args.head_layout != "tiled":
        case["name"] = case["name"] + "_" + args.head_layout
        case["head_layout"] = "borrowed (W read in place, row-major)"

    def refill_masks():
        masks.copy_(mask0.unsqueeze(0).expand_as(masks))
        torch.cuda.synchronize(dev)

    def step(i):
        mask = masks[i % n_masks]
        if B == 1:
            ctx.step(hidden, mask.reshape(N), case["tau"], case["budget"], commit[0], token[0], stats[0])
        else:
            ctx.step_batched(hidden, mask, case["tau"], case["budget"], commit, token, stats)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    def reduce_max(x):
        if world == 1:
            return x
        import torch.distributed as dist
        t = torch.tensor([x], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    refill_masks()
    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize(dev)
    st = [rpd.stats_dict(stats[b].cpu()) for b in range(B)]
    assert all(x["status"] == 0 for x in st), st
    extra_bytes = 0.0
    if args.projection != "all":
        # Lazy projection: the work is data dependent - the rows actually projected (FLOPs and
        # hidden-row bytes); the algorithmic bytes count the head once, and a second head
        # stream (when the band is not empty) is reported as extra traffic.
        nmt = sum(int(torch.count_nonzero(m)) for m in case["mask"].reshape(-1, N))
        rows_done = st[0]["n_rows"]
        passes = 1 if rows_done in (nmt, K * nmt) else 2
        flops = 2.0 * rows_done * d * V
        bytes_ = 2.0 * V * d + 2.0 * rows_done * d
        extra_bytes = (passes - 1) * 2.0 * V * d
        case["name"] = case["name"] + "_" + args.projection
        case["lazy_rows"] = rows_done
        case["lazy_passes"] = passes

    # Timed pass 1: the step time (no per-kernel events, which would serialise the
    # programmatic-dependent-launch overlap between the step's kernels).
    refill_masks()
    barrier()
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.steps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    barrier()
    ms_local = e0.elapsed_time(e1)
    # Timed pass 2: the same K steps with CUDA events around every launch on the context's
    # stream, for per-kernel durations (the roofline of the dominant kernel).
    refill_masks()
    ctx.kernel_times(reset=True)
    ctx.profile(True)
    for i in range(args.steps):
        step(i)
    torch.cuda.synchronize(dev)
    ctx.profile(False)
    clocks = sampler.stop() if sampler else None
    ktimes = ctx.kernel_times(reset=True)
    ms_total, ms_step, steps_s = aggregate_timing(ms_local, args.steps, world, reduce_max)

    # ---------------------------------------------------------------- end to end (host buffers)
    e2e = None
    if not args.no_e2e and B == 1:
        e2e = measure_e2e(ctx, case, args, world, barrier, reduce_max)

    if rank != 0:
        ctx.close()
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    ctx.close()
    trajectory = None
    if (not args.no_trajectory and world == 1 and args.workload == "llada_first_step"
            and not args.masked and not args.window and not args.block):
        # The decode trajectory at the same head shape (the head of this workload), every
        # layer projected and the projection chosen per step on the device.
        trajectory = trajectory_runs(case["W"], case["g"], ["all", "auto"], graph=True, warm=1,
                                     tiling=args.tiling)
        trajectory["device_loop"] = device_loop_runs(case["W"], case["g"])
    emit(args, case, R, flops, bytes_, ms_step, steps_s, ktimes, clocks, e2e,
         st[0] if B == 1 else st, world, extra_bytes=extra_bytes, trajectory=trajectory)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def measure_e2e(ctx, case, args, world, barrier, reduce_max):
    """Same step through rpd_step_host: inputs in pinned host memory (the step reads the masked
    positions' hidden rows across the host link; mask and canvas are copied in), results read
    back, every step inside the timed region."""
    N = case["N"]
    hid_h = case["hidden"].reshape(case["K"], N, case["d"]).contiguous().pin_memory()
    mask_h0 = case["mask"].reshape(N).clone()
    mask_h = mask_h0.clone().pin_memory()
    commit_h = torch.zeros(N, dtype=torch.uint8).pin_memory()
    token_h = torch.full((N,), -1, dtype=torch.int32).pin_memory()
    stats_h = torch.zeros(9, dtype=torch.int32).pin_memory()
    e2e_steps = max(3, min(args.steps, 200))
    for _ in range(2):
        mask_h.copy_(mask_h0)
        ctx.step_host(hid_h, mask_h, case["tau"], case["budget"], commit_h, token_h, stats_h)
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        mask_h.copy_(mask_h0)
        ctx.step_host(hid_h, mask_h, case["tau"], case["budget"], commit_h, token_h, stats_h)
    e2e_s = reduce_max(time.perf_counter() - t0)
    n_masked = int(mask_h0.sum())
    h2d = case["K"] * n_masked * case["d"] * 2 + N + N * 4   # masked rows, mask, canvas tokens
    d2h = N + N + N * 4 + 36                                  # mask, commits, tokens, stats
    return {"value": e2e_steps * world / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h,
            "api": "rpd_step_host (pinned host buffers; hidden rows of masked positions read in place)"}


def pick_peak(peaks, timed_s, clocks):
    """The measured peak that applies to a kernel timed over ``timed_s`` seconds: the burst
    figures when the timed region is shorter than a second or the clocks never showed the
    power cap, the sustained ones otherwise."""
    capped = bool(clocks) and "sw_power_cap" in clocks.get("reasons", [])
    sustained = timed_s >= 1.0 and capped
    return ("sustained" if sustained else "burst",
            peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"])


def emit(args, case, R, flops, bytes_, ms_step, steps_s, ktimes, clocks, e2e, st, world,
         extra_bytes=0.0, trajectory=None):
    K = case["K"]
    peaks = load_peaks()
    head_ms, head_n = ktimes["head_stats"]
    # head-statistics time per step (a lazy step runs one head pass per projection pass)
    head_avg_ms = head_ms / max(args.steps, 1)
    kind, tc_peak = pick_peak(peaks, args.steps * ms_step * 1e-3, clocks)
    t_tc = flops / (tc_peak * 1e12)
    t_hbm = bytes_ / (peaks["hbm_gbs"] * 1e9)
    if t_tc >= t_hbm:
        achieved = flops / (head_avg_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": tc_peak, "unit": "TFLOP/s",
                "frac": achieved / tc_peak, "traffic": None,
                "peak_kind": f"bf16 {kind}, of {peaks['source']}",
                "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"],
                "frac_of_nominal_dense_bf16": achieved / NOMINAL_BF16_TFLOPS}
    else:
        achieved = bytes_ / (head_avg_ms * 1e-3) / 1e9
        peak = peaks["hbm_gbs"]
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": None, "peak_kind": f"HBM copy, of {peaks['source']}",
                "frac_of_nominal_hbm": achieved / NOMINAL_HBM_GBS}
    step_roof = max(t_tc, t_hbm) / (ms_step * 1e-3)
    if roof["frac"] > 1.0:
        # the denominators are measured rates (a cuBLAS GEMM, a copy kernel), not hardware
        # limits: a kernel can exceed them a little, far more would mean skipped work
        roof["above_measured_peak"] = True
    roof["traffic"] = HEAD_TRAFFIC.get((case["name"], head_source_hash()))
    roof["algorithmic_bytes"] = bytes_
    roof["algorithmic_flops"] = flops
    if extra_bytes:
        # lazy projection: the second pass streams the head again; that is traffic beyond the
        # step's algorithmic bytes (the head once plus the projected rows)
        roof["extra_head_stream_bytes"] = extra_bytes

    cpu = None
    if not args.no_cpu_baseline and case.get("B", 1) == 1 and "block" not in case["rule"]:
        cpu = cpu_baseline(case, R, args)

    out = {
        "metric": METRIC, "value": steps_s, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_dict(case, R),
        "rows_per_s": steps_s * R,
        "roofline": roof,
        "step_roofline_frac": step_roof,
        "kernels_ms": {k: v[0] / max(args.steps, 1) for k, v in ktimes.items()},
        "kernel_timing": "per step; second timed pass of the same steps with CUDA events around each launch",
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches_per_step(case, args) * args.steps,
        "clocks": clocks,
        "last_step_stats": st,
    }
    if trajectory is not None:
        out["trajectory"] = trajectory
    print(json.dumps(out))


def cpu_baseline(case, R, args):
    """The oracle on a bounded sample of the workload (its first positions): the rate with one
    BLAS thread (the plain single-threaded oracle) and with every host core's BLAS threads."""
    pos = args.cpu_positions
    dt = oracle_step_seconds(case, pos)
    rows = case["K"] * pos
    multi = {"value": rows / dt / R, "unit": UNIT, "cores": blas_threads(), "rows_per_s": rows / dt,
             "seconds": dt}
    single = single_thread_oracle_rate(pos)
    if single is None:
        return dict(multi, kind="oracle", single_thread=None,
                    sample=f"oracle step over the first {pos} of {case['N']} masked positions "
                           f"({rows} rows, full V and d) with {multi['cores']} BLAS threads took "
                           f"{dt:.1f} s; rows/s scaled to the {R}-row step (single-thread run failed)")
    r1, dt1, thr1 = single
    return {"value": r1 / R, "unit": UNIT, "cores": thr1, "kind": "oracle", "rows_per_s": r1,
            "sample": f"oracle step over the first {pos} of {case['N']} masked positions ({rows} rows, "
                      f"full V and d, fp64 logits) with one BLAS thread took {dt1:.1f} s; rows/s "
                      f"scaled to the {R}-row step",
            "host_cores": os.cpu_count(),
            "multi_thread": dict(multi, sample=f"the same sample with {multi['cores']} BLAS threads "
                                               f"took {dt:.1f} s")}


def trajectory_runs(W, g, projections, graph=True, warm=1, tiling="auto"):
    """The decode trajectory at the LLaDA-8B head shape (N=256, K=4): up to 64 steps on one
    canvas; before each step the hidden states are regenerated from the seed for the current
    mask (context resolves left to right), the step's commits feed the next mask, and the run
    stops once at most 2% of the canvas is masked.  Each step is timed on the device with CUDA
    events around it (graph replay of the captured step when ``graph``); inputs are copied in
    before the events.  Per step the roofline time is max(FLOPs of the rows actually projected
    / tensor peak, (head once + those rows) / HBM peak).  Returns one summary per projection."""
    import paper_2609_36452_gb300 as rpd
    import workloads as WL
    dev = torch.device("cuda:0")
    K, N = 4, 256
    V, d = W.shape
    Wd, gd = W.to(dev), g.to(dev)
    gen = torch.Generator().manual_seed(4004)
    targets = torch.randint(0, V, (N,), generator=gen)
    peaks = load_peaks()
    hidden_d = torch.empty(K, N, d, dtype=torch.bfloat16, device=dev)
    mask_d = torch.empty(N, dtype=torch.uint8, device=dev)
    commit = torch.zeros(N, dtype=torch.uint8, device=dev)
    token = torch.full((N,), -1, dtype=torch.int32, device=dev)
    stats = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
    cache = {}
    results = {}
    for projection in projections:
        ctx = rpd.Rpd(d, V, K, 1e-6)
        ctx.set_head(Wd, gd)
        ctx.set_profile("llada")
        stream = torch.cuda.current_stream(dev)
        ctx.set_stream(stream)
        ctx.reserve(1, N)
        ctx.set_projection(projection)
        ctx.set_head_tiling(tiling)
        g_step = None
        if graph:
            mask_d.fill_(1)
            hidden_d.zero_()
            ctx.step(hidden_d, mask_d, 0.9, 1.0, commit, token, stats)  # configures the kernels
            torch.cuda.synchronize(dev)
            g_step = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_step):
                ctx.set_stream(torch.cuda.current_stream(dev))
                ctx.step(hidden_d, mask_d, 0.9, 1.0, commit, token, stats)
            ctx.set_stream(stream)

        def one_run():
            mask = torch.ones(N, dtype=torch.uint8)
            steps = []
            for t in range(64):
                key = (t, bytes(mask.numpy()))
                if key not in cache:
                    cache[key] = WL.trajectory_hidden(W, K, N, seed=4, step=t, mask=mask,
                                                      targets=targets).hidden.pin_memory()
                hidden_d.copy_(cache[key])
                mask_d.copy_(mask)
                torch.cuda.synchronize(dev)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                if g_step is not None:
                    g_step.replay()
                else:
                    ctx.step(hidden_d, mask_d, 0.9, 1.0, commit, token, stats)
                e1.record(stream)
                torch.cuda.synchronize(dev)
                nm = int(mask.sum())
                st = rpd.stats_dict(stats.cpu())
                assert st["status"] == 0 and st["n_masked"] == nm, st
                ms = e0.elapsed_time(e1)
                R = st["n_rows"]  # rows actually projected (lazy: data dependent)
                passes = 1 if R in (nm, K * nm) else 2
                roof_s = max(2.0 * R * d * V / (peaks["bf16_tflops"] * 1e12),
                             (2.0 * V * d + 2.0 * R * d) / (peaks["hbm_gbs"] * 1e9))
                steps.append({"t": t, "masked": nm, "committed": st["n_committed"], "rows": R,
                              "head_streams": passes, "ms": round(ms, 5),
                              "roofline_ms": round(roof_s * 1e3, 5),
                              "frac": round(roof_s * 1e3 / ms, 4)})
                mask = mask_d.cpu()
                if int(mask.sum()) <= 0.02 * N:
                    break
            return steps, int(mask.sum())

        for _ in range(warm):
            one_run()
        steps, remaining = one_run()
        ctx.close()
        total_ms = sum(x["ms"] for x in steps)
        roof_ms = sum(x["roofline_ms"] for x in steps)
        big = [x["frac"] for x in steps if x["rows"] >= 100]
        results[projection] = {
            "steps": len(steps), "total_ms": round(total_ms, 4),
            "steps_per_s": len(steps) / (total_ms / 1e3),
            "roofline_frac": roof_ms / total_ms,
            "min_frac_rows_ge_100": min(big) if big else None,
            "remaining_masked": remaining,
            "per_step": steps,
        }
    return {"workload": "llada_trajectory (N=256, K=4, d=4096, V=126464; steps until <= 2% "
                        "masked; hidden states regenerated per step from the seed)",
            "timing": ("CUDA graph replay of one step, " if graph else "") +
                      "CUDA events around each step, inputs copied in before the events",
            "roofline": "per step max(2*R*d*V / bf16 burst peak, (2*V*d + 2*R*d) / HBM peak), "
                        "R = rows actually projected; aggregate = sum of roofline times / sum of times",
            "peaks": {"bf16_tflops": peaks["bf16_tflops"], "hbm_gbs": peaks["hbm_gbs"],
                      "source": peaks["source"]},
            **results}


def device_loop_runs(W, g, repeats=3):
    """The LLaDA decode trajectory (N=256, K=4) with the decoding loop on the device: a
    stand-in for the backbone's forward pass - torch ops, captured as a CUDA graph, that rebuild
    the hidden states from the canvas before every step (the trajectory's generator: the signal
    of position p grows as the canvas left of p is committed; its noise is drawn once) - and the
    step repeat inside one graph launch until at most 2% of the canvas is masked
    (rpd_build_decode_loop).  Timed with CUDA events around one launch.  The same forward pass
    and step, replayed from the host with a read of the masked count after every step, are
    timed beside it: the difference is what returning to the host between steps costs."""
    import paper_2609_36452_gb300 as rpd
    import workloads as WL
    dev = torch.device("cuda:0")
    K, N = 4, 256
    V, d = W.shape
    gen = torch.Generator().manual_seed(4004)
    targets = torch.randint(0, V, (N,), generator=gen)
    flip = torch.randperm(N, generator=gen)[: N // 10]
    alt = (targets[flip] + torch.randint(1, V, (flip.numel(),), generator=gen)) % V
    wt = W[targets].float()
    wt = wt / wt.norm(dim=1, keepdim=True)
    wf = wt.clone()
    wf[flip] = W[alt].float() / W[alt].float().norm(dim=1, keepdim=True)
    dirs = torch.stack([wf if k == K - 2 else wt for k in range(K)]).to(dev)
    noise = torch.randn(K, N, d, generator=gen).to(dev)
    a = WL.layer_ramp(K).to(dev)
    base_b = WL.u_profile(N, 0.3, 4.0).to(dev)
    sigma = WL.DEFAULT_KAPPA * math.sqrt(d)
    pos = torch.arange(N, device=dev)
    denom = pos.clamp_min(1).float()
    hidden = torch.empty(K, N, d, dtype=torch.bfloat16, device=dev)
    mask = torch.ones(N, dtype=torch.uint8, device=dev)
    commit = torch.zeros(N, dtype=torch.uint8, device=dev)
    token = torch.full((N,), -1, dtype=torch.int32, device=dev)
    stats = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
    steps = torch.zeros(1, dtype=torch.int32, device=dev)

    def forward():
        committed = (mask == 0).float()
        before = torch.cumsum(committed, 0) - committed
        f = torch.where(pos > 0, before / denom, torch.ones_like(before))
        b = base_b + (4.0 - base_b).clamp_min(0) * f.pow(8)
        hidden.copy_((a[:, None, None] * sigma * b[None, :, None] * dirs + noise).to(torch.bfloat16))

    stream = torch.cuda.current_stream(dev)
    ctx = rpd.Rpd(d, V, K, 1e-6)
    ctx.set_stream(stream)
    ctx.set_head(W.to(dev), g.to(dev))
    ctx.set_profile("llada")
    ctx.reserve(1, N)
    try:
        fwd_graph = torch.cuda.CUDAGraph(keep_graph=True)
    except TypeError:
        return {"unavailable": "this PyTorch cannot hand out a captured graph (keep_graph)"}
    forward()
    with torch.cuda.graph(fwd_graph):
        forward()
    fwd_graph.instantiate()
    # the step alone, captured for the host-driven replay
    step_graph = torch.cuda.CUDAGraph()
    mask.fill_(1)
    ctx.step(hidden, mask, 0.9, 1.0, commit, token, stats)
    torch.cuda.synchronize(dev)
    with torch.cuda.graph(step_graph):
        ctx.set_stream(torch.cuda.current_stream(dev))
        ctx.step(hidden, mask, 0.9, 1.0, commit, token, stats)
    ctx.set_stream(stream)
    loop = ctx.build_decode_loop(hidden, mask, 0.9, 1.0, commit, token, stats, steps,
                                 stop_frac=0.02, max_steps=64, forward=fwd_graph)
    dev_ms, host_ms = [], []
    dev_steps = host_steps = 0
    for _ in range(repeats + 1):
        mask.fill_(1)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        loop.launch(stream)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        dev_ms.append(e0.elapsed_time(e1))
        dev_steps = int(steps.item())
        mask.fill_(1)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        n = 0
        while True:
            fwd_graph.replay()
            step_graph.replay()
            n += 1
            st = rpd.stats_dict(stats.cpu())  # the host reads the step's result
            if st["status"] != 0 or st["n_masked"] - st["n_committed"] <= int(0.02 * N) or n >= 64:
                break
        e1.record(stream)
        torch.cuda.synchronize(dev)
        host_ms.append(e0.elapsed_time(e1))
        host_steps = n
    loop.close()
    ctx.close()
    dev_t, host_t = sorted(dev_ms[1:])[len(dev_ms[1:]) // 2], sorted(host_ms[1:])[len(host_ms[1:]) // 2]
    return {"workload": "llada_trajectory_device_loop (N=256, K=4, d=4096, V=126464; forward "
                        "stand-in rebuilds the hidden states from the canvas on the device)",
            "steps": dev_steps, "total_ms": round(dev_t, 4), "steps_per_s": dev_steps / (dev_t / 1e3),
            "host_loop": {"steps": host_steps, "total_ms": round(host_t, 4),
                          "timing": "forward and step graph replays, host read of the step's "
                                    "statistics after every step"},
            "timing": f"median of {repeats} launches, CUDA events around one launch"}


def run_trajectory(args):
    """The decode trajectory alone (one projection, ``--projection``), as one JSON line."""
    import workloads as WL
    torch.cuda.set_device(torch.device("cuda:0"))
    W, g = WL.make_head(WL.LLADA_V, WL.LLADA_D, seed=2)
    out = trajectory_runs(W, g, [args.projection], graph=args.graph,
                          warm=max(1, args.warmup // 10), tiling=args.tiling)
    out["metric"] = METRIC
    out["unit"] = UNIT
    print(json.dumps(out))


def run_vocab_parallel(args):
    """The LLaDA first step with the LM head split over the ranks (rank r holds slice r of the
    vocabulary): per step every rank projects its slice, one NCCL all-gather moves 16 bytes per
    projected row and rank, and every rank merges the slices and commits.  Strong scaling (the
    same step on every N); at N = 1 the single slice is the whole head.  Timed like run_rpd."""
    import torch.distributed as dist

    import paper_2609_36452_gb300 as rpd
    from paper_2609_36452_gb300.vocab_parallel import shard_bounds, sharded_step
    rank, world, local = dist_env()
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
    os.environ.setdefault("MASTER_PORT", "29517")
    dist.init_process_group("nccl", rank=rank, world_size=world, device_id=dev)
    case = make_workload(0)  # every rank runs the same canvas
    K, N, d, V = case["K"], case["N"], case["d"], case["V"]
    v0, v1 = shard_bounds(V, world, rank)
    W = case["W"][v0:v1].contiguous().to(dev)
    g = case["g"].to(dev)
    hidden = case["hidden"].to(dev).contiguous()
    mask0 = case["mask"].to(dev)
    ctx = rpd.Rpd(d, v1 - v0, K, case["eps"])
    ctx.set_head(W, g)
    ctx.set_vocab_shard(v0, V)
    ctx.set_profile(case["rule"])
    stream = torch.cuda.current_stream(dev)
    ctx.set_stream(stream)
    ctx.reserve(1, N)
    n_masks = max(args.steps, args.warmup)
    masks = mask0.unsqueeze(0).repeat(n_masks, 1).contiguous()
    commit = torch.zeros(N, dtype=torch.uint8, device=dev)
    token = torch.full((N,), -1, dtype=torch.int32, device=dev)
    stats = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
    partials = torch.empty(K, N, 4, dtype=torch.float32, device=dev)
    gathered = torch.empty(world, K, N, 4, dtype=torch.float32, device=dev)

    def steps(n):
        for i in range(n):
            sharded_step(ctx, hidden, masks[i % n_masks], case["tau"], case["budget"], commit, token,
                         stats, partials=partials, gathered=gathered)

    masks.copy_(mask0.unsqueeze(0).expand_as(masks))
    steps(args.warmup)
    torch.cuda.synchronize(dev)
    assert rpd.stats_dict(stats.cpu())["status"] == 0
    masks.copy_(mask0.unsqueeze(0).expand_as(masks))
    dist.barrier()
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    steps(args.steps)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    dist.barrier()
    t = torch.tensor([e0.elapsed_time(e1)], device=dev, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    ms_step = float(t.item()) / args.steps
    R = rows_of(case)
    if rank == 0:
        peaks = load_peaks()
        roof = max(2.0 * R * d * V / (peaks["bf16_tflops"] * 1e12),
                   (2.0 * V * d + 2.0 * R * d) / (peaks["hbm_gbs"] * 1e9))
        print(json.dumps({
            "metric": METRIC, "value": 1e3 / ms_step, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": dict(config_dict(case, R), workload="llada_first_step_vocab_parallel",
                           parallelism=f"vocabulary slices over {world} GPUs, NCCL all-gather of "
                                       f"{16 * R} bytes per rank and step"),
            "rows_per_s": R * 1e3 / ms_step,
            "step_roofline_frac_whole_job": roof / (ms_step * 1e-3) / world,
            "gpu_launches": 7 * args.steps}))
    ctx.close()
    dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["rpd", "reference"], default="rpd")
    ap.add_argument("--workload", choices=["llada_first_step", "dream_mid_decode", "batched_serving",
                                           "trajectory"], default="llada_first_step")
    ap.add_argument("--block", action="store_true", help="RPD-block rule (blocks of 32)")
    ap.add_argument("--graph", action="store_true",
                    help="trajectory: replay each step from a captured CUDA graph")
    ap.add_argument("--projection", choices=["all", "lazy", "auto"], default="all",
                    help="window layers projected: all (the step as defined), lazy (earlier "
                         "layers only for band positions), auto (chosen per step on the device)")
    ap.add_argument("--head-layout", choices=["tiled", "borrowed"], default="tiled",
                    help="how the head kernel reads W: the context's tiled copy (default) or the "
                         "caller's row-major tensor in place")
    ap.add_argument("--tiling", choices=["auto", "pair", "rows_n"], default="auto",
                    help="head contraction tiling (default: chosen per pass on the device)")
    ap.add_argument("--cpu-positions", type=int, default=16,
                    help="positions of the oracle sample timed for cpu_baseline")
    ap.add_argument("--vocab-parallel", action="store_true",
                    help="LLaDA first step with the LM head split over the ranks (NCCL all-gather)")
    ap.add_argument("--no-trajectory", action="store_true",
                    help="leave the decode-trajectory object out of the default line")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--window", type=int, default=0,
                    help="LLaDA first step: project this many final layers (default 4; the "
                         "paper's LLaDA window is 16)")
    ap.add_argument("--masked", type=int, default=0,
                    help="keep only the last N canvas positions masked (head-streaming regime)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.vocab_parallel:
        run_vocab_parallel(args)
    elif args.workload == "trajectory":
        run_trajectory(args)
    else:
        run_rpd(args)


if __name__ == "__main__":
    main()

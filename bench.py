#!/usr/bin/env python
"""Benchmark of the GNMR per-step monitor on GB300.

One step = one gnmr_step over one full synthetic gradient arena: every unit's
L2 norm, Algorithm 1, the combined risk, Top_maxO with the lock bookkeeping
and the mask write (one kernel launch).  The default workload is the
LLaMA-2-13B layout: 40 layers x 7 linears = 280 bf16 units, 12.69 G elements
(25.38 GB) per step, larger than L2, so no flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gnmr|reference]

Prints one JSON line (rank 0).  Under torchrun (N > 1) each rank runs an
independent replica on its own GPU (the monitor has no exchange step on one
replica); time is the max over ranks and `value` counts every rank's bytes.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "GNMR step µs & grad GB/s (% HBM peak), LLaMA-2-13B 280-unit layout"
FALLBACK_HBM_GBS = 6800.0
PER_WORKLOADS = ("tiny", "llama2-1.3b", "llama2-13b", "moe", "aq-stress")
L2_BYTES = 129e6


def parse_args(argv=None):
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["gnmr", "reference"], default="gnmr")
    p.add_argument("--kernel", choices=["step", "actuator", "static-norms"], default="step",
                   help="step: the GNMR monitor (headline); actuator: the fake-quant actuator; "
                        "static-norms: the allocation-free per-unit norms entry point")
    p.add_argument("--tokens", type=int, default=4096, help="tokens per microbatch (actuator)")
    p.add_argument("--workload", default="llama2-13b")
    p.add_argument("--group", default="tensor", choices=["tensor", "block", "expert"],
                   help="unit granularity: one per tensor, per transformer block, per MoE expert")
    p.add_argument("--shrink", type=int, default=1,
                   help="divide matrix dims (small case for profiler captures)")
    p.add_argument("--arenas", type=int, default=2, help="distinct step arenas cycled")
    p.add_argument("--trace-steps", action="store_true",
                   help="time the workload's own consecutive trace steps: a fresh monitor runs the "
                        "steps before them untimed, every warm-up and timed step has its own arena "
                        "(they must all fit in device memory), and one untimed pass over those "
                        "arenas from the same state precedes the warm-up")
    p.add_argument("--e2e-steps", type=int, default=3)
    p.add_argument("--flush-l2", action="store_true",
                   help="write 512 MB before every timed step (outside its events)")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--graph", action="store_true",
                   help="capture the K timed steps (K gnmr_step launches) in one CUDA graph and "
                        "replay it: no host gaps between steps")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-sparsity", action="store_true",
                   help="skip the untimed pass over the trace that measures trigger sparsity")
    p.add_argument("--cpu-sample-units", type=int, default=0,
                   help="units in the CPU-oracle sample (0 = all: one full step)")
    p.add_argument("--ref-sample-units", type=int, default=0,
                   help="units per step of the reference arm (0 = every unit: the full step)")
    p.add_argument("--no-per-workload", action="store_true",
                   help="skip the per-workload records (every workload's own trace steps)")
    p.add_argument("--per-workload", default=",".join(PER_WORKLOADS),
                   help="comma-separated workloads for the per-workload records")
    args = p.parse_args(argv)
    if args.graph and args.flush_l2:
        p.error("--graph times back-to-back steps; it does not combine with --flush-l2")
    return args


# ---------------------------------------------------------------------------
# distributed helpers (replicas only)
# ---------------------------------------------------------------------------

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Max of a per-rank float over all ranks (identity for one rank)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def throughput_gbs(world: int, bytes_per_step: int, steps: int, max_ms: float) -> float:
    """Whole-job GB/s: every rank's gradient bytes over the slowest rank's time."""
    return world * bytes_per_step * steps / (max_ms / 1e3) / 1e9


def barrier(world: int, device=None):
    if world > 1:
        import torch.distributed as dist
        if device is not None and dist.get_backend() == "nccl":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 20):
        self.rows = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(gpu_index), "-lms", str(interval_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=5)

    def summary(self, t0: float, t1: float) -> dict:
        inside = [r for ts, r in self.rows if t0 <= ts <= t1]
        window = "timed region"
        if not inside:
            inside = [r for ts, r in self.rows if t0 - 0.5 <= ts <= t1 + 0.5]
            window = "within 0.5 s of the timed region"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi gave no sample"}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[2]) for r in inside if num(r[2]) is not None]
        mx = [num(r[3]) for r in inside if num(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i in range(4)
                          if len(r) > 6 + i and r[6 + i].lower().startswith("active")})
        power = [num(r[4]) for r in inside if num(r[4]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(inside), "window": window,
                "power_w_max": max(power) if power else None}


STEP_KERNEL_SOURCES = [os.path.join(ROOT, "paper_2606_00539_gb300", "csrc", f)
                       for f in ("gnmr_kernels.cu", "gnmr_stream.cuh", "gnmr_internal.h")]


def kernel_source_hash(paths) -> str:
    """First 16 hex digits of the sha256 of the concatenated source files with
    comments removed and whitespace collapsed: an edit to a comment leaves the
    compiled kernel, and so its profile, unchanged."""
    import hashlib
    import re
    h = hashlib.sha256()
    for path in paths:
        with open(path, encoding="utf-8") as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(paths, workload: str = "llama2-13b"):
    """DRAM bytes per launch of `workload`'s step from the committed ncu
    record, or None if there is none or the kernel's sources have changed
    since its counters were taken."""
    try:
        with open(os.path.join(ROOT, "profiles", "gnmr_step_kernel_traffic.json")) as f:
            rec = json.load(f)["records"][workload]
        h = kernel_source_hash(paths)
    except (OSError, KeyError, TypeError, ValueError):
        return None
    if rec.get("kernel_source_sha256_16") != h:
        return None
    return int(rec["traffic_bytes_per_launch"])


def grid_text(info) -> str:
    """Launch geometry of a handle, from gnmr_get_info."""
    if info["loop_shape"] == 2:
        return (f"{info['num_ctas']} CTAs x {info['threads_per_cta']} threads, {info['num_runs']} runs "
                f"taken dynamically by {info['num_warps']} warps, large-unit loop shape")
    return (f"{info['num_ctas']} CTAs x {info['threads_per_cta']} threads, {info['num_warps']} warp runs, "
            f"small-unit loop shape")


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# ---------------------------------------------------------------------------
# CPU baseline: the oracle on a bounded sample of the same workload
# ---------------------------------------------------------------------------

def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_oracle_rate(view, w, units, reps: int = 1, threads: int = 0):
    """Times the oracle (norms of `units` + Algorithms 1-2 over them) and
    returns (GB/s, threads, seconds per rep); threads = 0: every host core."""
    import oracle
    off = w.offsets[units]
    ln = w.lengths[units]
    threads = min(threads or host_cores(), len(units))
    ctl = oracle.Controller(len(units), **dict(w.controller_kwargs(),
                                               recoverable=w.recoverable[units]))
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        n = oracle.unit_norms_threaded(view, off, ln, threads)
        ctl.step(n)
        times.append(time.perf_counter() - t0)
    ctl.close()
    sec = statistics.median(times)
    nbytes = int(ln.sum()) * w.elem_bytes
    return nbytes / sec / 1e9, threads, sec


def workload_config(w, args, n_arenas: int, world: int) -> dict:
    """The `config` object both arms print: what the workload is, not how a
    kernel runs it (the same dict on the GPU arm and the reference arm)."""
    return {"workload": f"{w.name} ({w.num_units} units, {w.num_segments} tensors, "
                        f"{w.grad_elems} {w.dtype} "
                        f"elements{'' if args.shrink == 1 else f', dims / {args.shrink}'})",
            "bytes_per_step": w.grad_bytes,
            "arenas_cycled": args.warmup + args.steps if getattr(args, "trace_steps", False) else n_arenas,
            **({"trace_steps": list(trace_span(w, args))} if getattr(args, "trace_steps", False) else {}),
            "l2": ("L2 flushed before every step (512 MB write)" if getattr(args, "flush_l2", False)
                   else "inputs larger than L2 (no flush)" if w.grad_bytes > 2 * L2_BYTES
                   else "inputs fit in L2 (hot)"),
            "parallelism": "replicas" if world > 1 else "single GPU"}


# ---------------------------------------------------------------------------
# reference arm: the oracle on the host cores
# ---------------------------------------------------------------------------

HOST_BLOCK = 1 << 24


def host_arena(w, step: int, units, threads: int) -> np.ndarray:
    """A host copy of one arena of workload `w` (same packing: w.offsets,
    w.arena_elems) for the oracle, generated on the host cores without the
    GPU.  One seeded N(0, 1) block of 16 Mi values is tiled over every unit
    (starting at a unit-dependent position) and scaled by the power of two
    nearest the unit's scale at trace step `step` (0-based), which for these
    float formats is an exact integer add on the exponent field; a unit with
    scale 0 (an unrouted expert) is all zeros.  The oracle's cost does not
    depend on the values, only on the layout."""
    from concurrent.futures import ThreadPoolExecutor
    rng = np.random.default_rng([w.seed, 17, step])
    block = rng.standard_normal(HOST_BLOCK, dtype=np.float32)
    block[np.abs(block) < 1e-6] = 1e-6                       # keep every value normal
    if w.dtype == "bf16":
        u = block.view(np.uint32)
        u += ((u >> 16) & 1) + 0x7FFF                          # round to nearest even
        bits = (u >> 16).astype(np.uint16)
        out = np.zeros(w.arena_elems, np.uint16)
        shift, dt = 7, np.uint16
    else:
        bits = block.view(np.uint32).copy()
        out = np.zeros(w.arena_elems, np.float32)
        shift, dt = 23, np.uint32
    view = out.view(dt)
    scales = w.scales[step]

    def one(s):
        sc = float(scales[s])
        if sc == 0.0:
            return
        k = int(round(math.log2(sc)))
        off, n = int(w.offsets[s]), int(w.lengths[s])
        start = (s * 7919) % HOST_BLOCK
        pos = 0
        while pos < n:
            take = min(n - pos, HOST_BLOCK - start)
            dst = view[off + pos:off + pos + take]
            np.copyto(dst, bits[start:start + take])
            # |k| is small (log-normal scales, spikes up to 10^4), so no
            # exponent field over- or underflows
            if k > 0:
                np.add(dst, dt(k << shift), out=dst)
            elif k < 0:
                np.subtract(dst, dt(-k << shift), out=dst)
            pos += take
            start = 0

    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        list(ex.map(one, [int(s) for s in units]))
    return out


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    import oracle
    import workloads
    w = workloads.make(args.workload, shrink=args.shrink)
    k = args.ref_sample_units or w.num_units
    units = np.arange(min(k, w.num_units))
    off = w.offsets[units]
    ln = w.lengths[units]
    threads = min(host_cores(), len(units))
    n_arenas = max(1, args.arenas)
    # the trace steps the GPU arm cycles, generated on the host (untimed)
    arenas = [host_arena(w, (w.steps // 2 + i) % w.steps, units, host_cores()) for i in range(n_arenas)]
    ctl = oracle.Controller(len(units), **dict(w.controller_kwargs(),
                                               recoverable=w.recoverable[units]))
    for i in range(args.warmup):
        ctl.step(oracle.unit_norms_threaded(arenas[i % n_arenas], off, ln, threads))
    t0 = time.perf_counter()
    for i in range(args.steps):
        ctl.step(oracle.unit_norms_threaded(arenas[(args.warmup + i) % n_arenas], off, ln, threads))
    sec = (time.perf_counter() - t0) / max(args.steps, 1)
    ctl.close()
    nbytes = int(ln.sum()) * w.elem_bytes
    gbs = nbytes / sec / 1e9
    full = len(units) == w.num_units
    what = (f"every step the whole {w.num_units}-unit {w.name} layout" if full
            else f"units 0..{len(units) - 1} of the {w.num_units}-unit {w.name} layout")
    sample = (f"{what} ({nbytes / 1e9:.3f} GB of {w.grad_bytes / 1e9:.3f} GB per step): unit norms "
              f"on {threads} threads (contiguous unit groups of equal bytes, each unit summed "
              f"sequentially in double) + Algorithms 1-2; {n_arenas} host-generated arenas cycled")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(gbs, 4), "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(nbytes / (gbs * 1e9) * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": "synthetic",
        "config": workload_config(w, args, n_arenas, world),
        "cpu_baseline": {"value": round(gbs, 4), "unit": "GB/s", "cores": threads,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(gbs, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    if not full:
        line["note"] = "a sample of the layout's units: value is the sample's GB/s"
    print(json.dumps(line), flush=True)


def exceedance_counts(gnmr, dgnmr, recoverable, alpha_t: float, beta_t: float):
    """One step's contribution to the trigger-sparsity statistic of Table 3:
    among the recoverable units, how many have GNMR > alpha_t and how many
    Delta-GNMR > beta_t (the two thresholds of the combined risk, Sec. 3.3)."""
    rec = np.asarray(recoverable) != 0
    return (int(np.count_nonzero(rec & (np.asarray(gnmr) > alpha_t))),
            int(np.count_nonzero(rec & (np.asarray(dgnmr) > beta_t))))


def trigger_sparsity(w, filler, arena, dev) -> dict:
    """Table 3's statistic on the workload's synthetic trace: a fresh monitor
    runs steps 1..T of the trace (untimed, after the timed region) and the
    share of (recoverable unit, step) pairs over each threshold is counted,
    with the candidate and selected counts of Algorithm 2.  Table 11's two
    trigger statistics come with it: the promotion ratio (selected
    (unit, step) pairs over all of them) and the hit-maxO rate, read as the
    share of steps at which |A_t| reached the budget maxO."""
    import torch
    from paper_2606_00539_gb300 import Monitor
    mon = Monitor(w.offsets, w.lengths, device=dev.index, **w.monitor_kwargs())
    stats = mon.new_stats()
    mask = torch.empty(w.num_units, dtype=torch.uint8, device=dev)
    rec = np.asarray(w.recoverable, np.uint8)
    over_g = over_d = cand = sel = hit = 0
    try:
        for t in range(w.steps):
            filler.fill(arena, t)
            mon.step(arena, mask=mask, stats=stats)
            a_t = w.alpha[0] if t + 1 <= w.warmup_steps else w.alpha[1]
            b_t = w.beta[0] if t + 1 <= w.warmup_steps else w.beta[1]
            g, d = exceedance_counts(stats["gnmr"].cpu().numpy(), stats["dgnmr"].cpu().numpy(), rec, a_t, b_t)
            c = stats["counts"].cpu().tolist()
            over_g, over_d, cand, sel = over_g + g, over_d + d, cand + c[0], sel + c[1]
            hit += int(w.max_o > 0 and c[1] >= w.max_o)
    finally:
        mon.close()
    pairs = max(1, int(rec.sum()) * w.steps)
    return {"gnmr_over_alpha_pct": round(100.0 * over_g / pairs, 4),
            "dgnmr_over_beta_pct": round(100.0 * over_d / pairs, 4),
            "candidates_per_step": round(cand / w.steps, 2),
            "selected_per_step": round(sel / w.steps, 2),
            "selected_pct": round(100.0 * sel / pairs, 4),
            "promotion_ratio": round(sel / pairs, 6),
            "hit_max_o_rate": round(hit / w.steps, 4),
            "steps": w.steps, "recoverable_units": int(rec.sum()),
            "trace": "the workload's synthetic trace, steps 1..T, one fresh monitor, untimed"}


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def trace_span(w, args):
    """(first, last) trace step timed by --trace-steps (1-based)."""
    t0, k = trace_window(w.steps, args.steps, args.warmup)
    return t0, t0 + k - 1


def trace_window(trace_steps: int, k: int, w: int):
    """(first timed trace step, 1-based; number of timed steps): K steps in
    the middle of the trace, after at least W warm-up steps."""
    w = max(0, min(w, trace_steps - 1))
    k = max(1, min(k, trace_steps - w))
    t0 = max(w + 1, (trace_steps - k) // 2 + 1)
    return t0, min(k, trace_steps - t0 + 1)


def workload_record(name, k_steps, w_steps, dev, peak, sampler, budget_bytes):
    """workload_record_on with every allocation, fill, step and event on one
    stream, so their order is the order of the calls."""
    import torch
    stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        return workload_record_on(stream, name, k_steps, w_steps, dev, peak, sampler, budget_bytes)


def workload_record_on(stream, name, k_steps, w_steps, dev, peak, sampler, budget_bytes):
    """One workload's timing on its own trace: a fresh monitor runs trace
    steps 1..t0-1 (warm-up), its state is saved, and each timing pass
    restores it and runs trace steps t0..t0+K-1, so every pass makes the
    trace's own candidate pools and selections.  Arenas that fit in
    `budget_bytes` are all generated first (passes: back-to-back prepared
    calls with per-step events, one CUDA graph of the K calls, and, for
    arenas under 2 GB, an L2 flush (a 512 MB write) before every step, and an
    L2 clean (a 512 MB read, no dirty lines left) before every step; the graph
    pass reports the better of two timed replays); larger ones are
    regenerated between steps, outside each step's events, followed by a
    512 MB read so the step starts with no dirty or arena lines in L2."""
    import torch
    import workloads
    from paper_2606_00539_gb300 import Monitor

    w = workloads.make(name)
    filler = workloads.Filler(w, dev)
    t0, K = trace_window(w.steps, k_steps, w_steps)
    mon = Monitor(w.offsets, w.lengths, device=dev.index, **w.monitor_kwargs())
    info = mon.info()
    stats = mon.new_stats()
    counts = torch.zeros((K, 2), dtype=torch.int32, device=dev)
    mask = torch.empty(w.num_units, dtype=torch.uint8, device=dev)
    arena_bytes = w.arena_elems * w.elem_bytes
    distinct = K * arena_bytes <= budget_bytes
    rec = {"trace_steps": [t0, t0 + K - 1], "steps": K, "warmup_steps": t0 - 1,
           "units": w.num_units, "dtype": w.dtype, "bytes_per_step": w.grad_bytes,
           "grid": grid_text(info)}
    def fill(arena, i):
        filler.fill(arena, i)                       # on the current stream: `stream`

    # |C_t|, |A_t| of every trace step not timed: the warm-up steps here, the
    # steps after the timed window at the end
    trace_counts = torch.zeros((w.steps, 2), dtype=torch.int32, device=dev)
    scratch = filler.new_arena()
    for i in range(t0 - 1):                         # warm-up: trace steps 1..t0-1
        fill(scratch, i)
        mon.step(scratch, mask=mask, stats=dict(stats, counts=trace_counts[i]), stream=stream)
    blob = mon.get_state(stream)
    step_stats = [dict(stats, counts=counts[j]) for j in range(K)]
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    region = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    per_pass_counts = []

    def us(ms):
        return round(ms * 1e3, 1)

    if distinct:
        del scratch
        arenas = []
        for j in range(K):
            a = filler.new_arena()
            fill(a, t0 - 1 + j)
            arenas.append(a)
        calls = [mon.prepare_step(arenas[j], mask=mask, stats=step_stats[j], stream=stream) for j in range(K)]
        # untimed pass over the same steps: the first steps after the arenas
        # were generated ran up to ~10 % slower (measured), which no later pass shows
        mon.set_state(blob, stream)
        for j in range(K):
            calls[j]()
        stream.synchronize()
        # pass 1: back-to-back prepared calls (one C call per step, nothing
        # else on the host between them), timed as a region
        mon.set_state(blob, stream)
        wall0 = time.time()
        region[0].record(stream)
        t_host = time.perf_counter()
        for j in range(K):
            calls[j]()
        t_host = time.perf_counter() - t_host
        region[1].record(stream)
        stream.synchronize()
        per_pass_counts.append(counts.cpu().numpy().copy())
        rec["arenas"] = f"{K} distinct trace-step arenas, generated before timing"
        rec["us_per_step"] = us(region[0].elapsed_time(region[1]) / K)
        rec["host_us_per_call"] = round(t_host / K * 1e6, 1)
        # pass 1b: the same steps, each bracketed by its own event pair (the
        # kernel durations; the event records add host time between launches)
        mon.set_state(blob, stream)
        for j in range(K):
            ev[j][0].record(stream)
            calls[j]()
            ev[j][1].record(stream)
        stream.synchronize()
        per_ms = [a.elapsed_time(b) for a, b in ev]
        per_pass_counts.append(counts.cpu().numpy().copy())
        # pass 2: the K calls captured in one CUDA graph and replayed
        mon.set_state(blob, stream)
        graph = torch.cuda.CUDAGraph()
        stream.synchronize()
        with torch.cuda.graph(graph, stream=stream):
            for j in range(K):
                calls[j]()
        graph.replay()                               # untimed: the first replay uploads the graph
        g_runs = []
        for _ in range(2):                           # the better of two timed replays
            mon.set_state(blob, stream)
            torch.cuda.synchronize(dev)
            region[0].record(stream)
            graph.replay()
            region[1].record(stream)
            stream.synchronize()
            g_runs.append(region[0].elapsed_time(region[1]) / K)
            per_pass_counts.append(counts.cpu().numpy().copy())
        g_ms = min(g_runs)
        rec["graph_us_per_step"] = us(g_ms)
        rec["graph_gbs"] = round(w.grad_bytes / (g_ms / 1e3) / 1e9, 1)
        rec["graph_frac"] = round(w.grad_bytes / (g_ms / 1e3) / 1e9 / peak, 4)
        del graph
        # pass 3: L2 flushed (a 512 MB write) before every step, outside its events
        if arena_bytes < 2e9:
            flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
            mon.set_state(blob, stream)
            for j in range(K):
                flush.zero_()
                ev[j][0].record(stream)
                calls[j]()
                ev[j][1].record(stream)
            stream.synchronize()
            fl = [a.elapsed_time(b) for a, b in ev]
            per_pass_counts.append(counts.cpu().numpy().copy())
            rec["l2_flushed_us_mean"] = us(statistics.mean(fl))
            # the same with L2 emptied by a 512 MB read: no dirty lines left to
            # write back during the step, so this is the cost of cold state alone
            clean_out = torch.empty((), dtype=torch.int64, device=dev)
            mon.set_state(blob, stream)
            for j in range(K):
                torch.sum(flush, dim=0, dtype=torch.int64, out=clean_out)
                ev[j][0].record(stream)
                calls[j]()
                ev[j][1].record(stream)
            stream.synchronize()
            per_pass_counts.append(counts.cpu().numpy().copy())
            rec["l2_cleaned_us_mean"] = us(statistics.mean(a.elapsed_time(b) for a, b in ev))
            del flush, clean_out
        wall1 = time.time()
        del calls, arenas
    else:
        ring = [scratch, filler.new_arena()]
        clean = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
        clean_out = torch.empty((), dtype=torch.int64, device=dev)
        wall0 = time.time()
        for j in range(K):
            a = ring[j % 2]
            fill(a, t0 - 1 + j)
            torch.sum(clean, dim=0, dtype=torch.int64, out=clean_out)
            ev[j][0].record(stream)
            mon.step(a, mask=mask, stats=step_stats[j], stream=stream)
            ev[j][1].record(stream)
        stream.synchronize()
        wall1 = time.time()
        per_ms = [a.elapsed_time(b) for a, b in ev]
        per_pass_counts.append(counts.cpu().numpy().copy())
        rec["arenas"] = ("two arenas, each regenerated with the next trace step between steps (outside the "
                         "step's events), then a 512 MB read")
        rec["us_per_step"] = us(statistics.mean(per_ms))
        del ring, clean, clean_out
    # the rest of the trace (untimed), from the state the timed steps left
    if t0 + K - 1 < w.steps:
        scratch = filler.new_arena()
        for i in range(t0 + K - 1, w.steps):
            fill(scratch, i)
            mon.step(scratch, mask=mask, stats=dict(stats, counts=trace_counts[i]), stream=stream)
        del scratch
    mon.close()
    kern = statistics.mean(per_ms)
    c = per_pass_counts[0]
    whole = trace_counts.cpu().numpy()
    whole[t0 - 1:t0 - 1 + K] = c
    rec.update({
        "trace_candidates_mean": round(float(whole[:, 0].mean()), 1),
        "trace_selected_mean": round(float(whole[:, 1].mean()), 2),
        "trace_hit_max_o_rate": round(float(np.mean(whole[:, 1] >= w.max_o)), 4) if w.max_o > 0 else 0.0,
        "kernel_us_mean": us(kern), "kernel_us_median": us(statistics.median(per_ms)),
        "kernel_us_min": us(min(per_ms)), "kernel_us_max": us(max(per_ms)),
        "gbs": round(w.grad_bytes / (kern / 1e3) / 1e9, 1),
        "frac": round(w.grad_bytes / (kern / 1e3) / 1e9 / peak, 4),
        "candidates_mean": round(float(c[:, 0].mean()), 1), "candidates_max": int(c[:, 0].max()),
        "selected_mean": round(float(c[:, 1].mean()), 2), "max_o": w.max_o,
        "passes_agree": all(np.array_equal(c, x) for x in per_pass_counts[1:]),
        "traffic": profiled_traffic(STEP_KERNEL_SOURCES, w.name),
        "clocks": sampler.summary(wall0, wall1),
    })
    torch.cuda.synchronize(dev)
    torch.cuda.empty_cache()
    return rec


def per_workload_records(args, dev, peak, peak_kind) -> dict:
    """Every workload of --per-workload timed on its own trace steps (see
    workload_record); frac is GB/s over the kernel mean against the peak."""
    import torch
    names = [n for n in args.per_workload.split(",") if n]
    free, _ = torch.cuda.mem_get_info(dev)
    budget = 0.45 * free
    sampler = ClockSampler(dev.index)
    time.sleep(0.3)
    out = {"peak_gbs": peak, "peak_source": f"{peak_kind} hbm_gbs",
           "what": ("per workload: trace steps t0..t0+K-1 of its own synthetic trace after a fresh monitor "
                    "ran steps 1..t0-1; us_per_step = back-to-back prepared calls (distinct arenas) or the "
                    "kernel mean (regenerated arenas); host_us_per_call = host time of one prepared call; "
                    "kernel_us_* from per-step CUDA events; gbs and frac "
                    "from the kernel mean; candidates = |C_t| over the timed steps; trace_* = |C_t|, |A_t| "
                    "and the share of steps with |A_t| = maxO over all steps of the trace")}
    try:
        for n in names:
            out[n] = workload_record(n, args.steps, args.warmup, dev, peak, sampler, budget)
    finally:
        sampler.stop()
    return out


def run_gnmr(args):
    import torch
    import workloads
    from paper_2606_00539_gb300 import Monitor

    rank, local_rank, world = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)

    w = workloads.make(args.workload, shrink=args.shrink, seed=rank, group=args.group)
    filler = workloads.Filler(w, dev)
    mon = Monitor(w.offsets, w.lengths, device=local_rank, **w.monitor_kwargs())
    info = mon.info()
    stats = mon.new_stats()
    mask = torch.empty(w.num_units, dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(dev)
    arenas = []
    if args.trace_steps:
        # the trace's own steps: 1..first-1 untimed on one arena, then one
        # arena per warm-up and timed step
        t0, t1 = trace_span(w, args)
        if t1 - t0 + 1 != args.steps:
            raise SystemExit(f"--trace-steps: {w.name}'s trace has {w.steps} steps, too few for "
                             f"{args.warmup} + {args.steps}")
        first = t0 - args.warmup
        need = (args.warmup + args.steps) * w.arena_elems * w.elem_bytes
        if need > 0.8 * torch.cuda.mem_get_info(dev)[0]:
            raise SystemExit(f"--trace-steps: {need / 1e9:.1f} GB of arenas do not fit on the device")
        with torch.cuda.stream(stream):
            scratch = filler.new_arena()
            for i in range(first - 1):
                filler.fill(scratch, i)
                mon.step(scratch, mask=mask, stats=stats, stream=stream)
            del scratch
            for i in range(args.warmup + args.steps):
                a = filler.new_arena()
                filler.fill(a, first - 1 + i)
                arenas.append(a)
    else:
        for i in range(max(1, args.arenas)):
            # steps from the middle of the trace: spikes, ramps and locks are live
            a = filler.new_arena()
            filler.fill(a, (w.steps // 2 + i) % w.steps)
            arenas.append(a)
    n_arenas = len(arenas)
    torch.cuda.synchronize(dev)

    # one prepared gnmr_step call per arena: a step costs one C call on the host
    calls = [mon.prepare_step(a, mask=mask, stats=stats, stream=stream) for a in arenas]
    if args.trace_steps:
        # one untimed pass over every arena first, from the same controller
        # state: the first read of a freshly generated arena runs up to ~10 %
        # slower (measured), which no later read shows
        blob = mon.get_state(stream)
        for c in calls:
            c()
        mon.set_state(blob, stream)
    for i in range(args.warmup):
        calls[i % n_arenas]()
    stream.synchronize()

    graph = None
    if args.graph:
        # the captured steps run (and advance the controller) only when replayed
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for i in range(args.steps):
                calls[(args.warmup + i) % n_arenas]()
        blob = mon.get_state(stream) if args.trace_steps else None
        with torch.cuda.stream(stream):
            graph.replay()                # untimed: the first replay uploads the graph
        torch.cuda.synchronize(dev)
        if blob is not None:
            mon.set_state(blob, stream)   # the timed replay runs the same trace steps again
            torch.cuda.synchronize(dev)

    sampler = ClockSampler(local_rank)
    time.sleep(0.3)                       # let nvidia-smi start sampling
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    barrier(world, dev)
    torch.cuda.synchronize(dev)
    wall0 = time.time()
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev) if args.flush_l2 else None
    if graph is not None:
        t_start.record(stream)
        with torch.cuda.stream(stream):
            graph.replay()
        t_end.record(stream)
    else:
        t_start.record(stream)
        for i in range(args.steps):
            if flush is not None:
                with torch.cuda.stream(stream):
                    flush.zero_()
            ev[i][0].record(stream)
            calls[(args.warmup + i) % n_arenas]()
            ev[i][1].record(stream)
        t_end.record(stream)
    stream.synchronize()
    torch.cuda.synchronize(dev)
    wall1 = time.time()
    barrier(world, dev)
    sampler.stop()
    clocks = sampler.summary(wall0, wall1)

    if graph is not None:
        # back-to-back launches of one kernel: its mean duration is the region / K
        per_ms = [t_start.elapsed_time(t_end) / args.steps] * args.steps
    else:
        per_ms = [a.elapsed_time(b) for a, b in ev]
    # with flushes in the region, the step time is the sum of the steps' own events
    total_ms = sum(per_ms) if flush is not None else t_start.elapsed_time(t_end)
    max_ms = max_over_ranks(total_ms, world, dev)
    launches = args.steps                              # one kernel per gnmr_step

    gbytes = w.grad_bytes / 1e9
    value = throughput_gbs(world, w.grad_bytes, args.steps, max_ms)
    step_ms = max_ms / args.steps
    kern_ms = statistics.mean(per_ms)
    peak, peak_kind = measured_peaks()
    achieved = gbytes / (kern_ms / 1e3)
    traffic = profiled_traffic(STEP_KERNEL_SOURCES, w.name)

    # end to end through the public API with the step's input in pinned host
    # memory and its result read back to the host, every step inside the
    # timed region.  e2e: gnmr_step reads the host arena in place (its loads
    # cross the host link; no staging copy or device buffer).  e2e_staged: an
    # explicit host->device copy of the arena, then gnmr_step on the copy.
    e2e = None
    e2e_staged = None
    host = None
    if not args.no_e2e and args.e2e_steps > 0:
        why = None
        try:
            host = torch.empty(arenas[0].numel(), dtype=arenas[0].dtype, pin_memory=True)
            host.copy_(arenas[0])
            host_mask = torch.empty(w.num_units, dtype=torch.uint8, pin_memory=True)
        except RuntimeError as exc:
            why = str(exc).splitlines()[0]
            host = None
        # every rank takes the same branch: the timed loops below hold collectives
        if max_over_ranks(0.0 if why is None else 1.0, world, dev) > 0.0:
            e2e = {"value": None, "unit": "GB/s",
                   "error": why or "pinned host allocation failed on another rank"}
            host = None
        else:
            dst = arenas[-1]
            h2d = int(host.numel() * host.element_size())

            def timed(one_step):
                for i in range(args.e2e_steps + 1):
                    if i == 1:
                        torch.cuda.synchronize(dev)
                        e0 = torch.cuda.Event(enable_timing=True)
                        e1 = torch.cuda.Event(enable_timing=True)
                        e0.record(stream)
                    with torch.cuda.stream(stream):
                        one_step()
                        host_mask.copy_(mask, non_blocking=True)
                    stream.synchronize()
                e1.record(stream)
                stream.synchronize()
                return max_over_ranks(e0.elapsed_time(e1) / args.e2e_steps, world, dev)

            def staged():
                dst.copy_(host, non_blocking=True)
                mon.step(dst, mask=mask, stream=stream)

            try:
                ms = timed(lambda: mon.step(host, mask=mask, stream=stream))
                e2e = {"value": round(world * gbytes / (ms / 1e3), 3), "unit": "GB/s",
                       "ms_per_step": round(ms, 3), "h2d_bytes_per_step": h2d,
                       "d2h_bytes_per_step": int(w.num_units), "steps": args.e2e_steps,
                       "path": "gnmr_step reading the pinned host arena in place, mask -> pinned host"}
                ms = timed(staged)
                e2e_staged = {"value": round(world * gbytes / (ms / 1e3), 3), "unit": "GB/s",
                              "ms_per_step": round(ms, 3), "h2d_bytes_per_step": h2d,
                              "d2h_bytes_per_step": int(w.num_units), "steps": args.e2e_steps,
                              "path": "pinned host arena -> device copy, gnmr_step, mask -> pinned host"}
            except RuntimeError as exc:
                if world > 1:
                    raise          # the other ranks wait in a collective: fail loudly, not hang
                e2e = {"value": None, "unit": "GB/s", "error": str(exc).splitlines()[0]}
                host = None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:     # the host baseline: N = 1 only
        k = args.cpu_sample_units or w.num_units
        units = np.arange(min(k, w.num_units))
        hi = int(w.offsets[units[-1]] + w.lengths[units[-1]])
        src = host[:hi] if host is not None else arenas[0][:hi].cpu()
        view = src.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16" else src.numpy()
        rate, threads, sec = cpu_oracle_rate(view, w, units)
        what = ("one full step" if len(units) == w.num_units
                else f"units 0..{len(units) - 1} of {w.num_units}")
        cpu = {"value": round(rate, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
               "sample": (f"{what} ({int(w.lengths[units].sum()) * w.elem_bytes / 1e9:.3f} GB of "
                          f"{gbytes:.3f} GB per step): unit norms + Algorithms 1-2, "
                          f"{sec:.2f} s wall on {threads} threads (contiguous unit groups of "
                          f"equal bytes, each unit summed sequentially in double)")}
        # one thread on a bounded prefix of the same layout (about 1.3 GB)
        cum = np.cumsum(w.lengths[units]) * w.elem_bytes
        one = units[:max(1, int(np.searchsorted(cum, 1.3e9)) + 1)]
        rate1, _, sec1 = cpu_oracle_rate(view, w, one, threads=1)
        cpu["single_thread"] = {
            "value": round(rate1, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": (f"units 0..{len(one) - 1} of {w.num_units} "
                       f"({int(w.lengths[one].sum()) * w.elem_bytes / 1e9:.3f} GB): unit norms + "
                       f"Algorithms 1-2 on one thread, {sec1:.2f} s wall")}
    del host

    sparsity = None
    if rank == 0 and not args.no_sparsity:
        sparsity = trigger_sparsity(w, filler, arenas[0], dev)

    per_workload = None
    if rank == 0 and world == 1 and not args.no_per_workload and args.shrink == 1 and args.group == "tensor":
        del calls, arenas, graph
        mon.close()
        torch.cuda.synchronize(dev)
        torch.cuda.empty_cache()
        per_workload = per_workload_records(args, dev, peak, peak_kind)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_ms, 4),
            "us_per_step": round(step_ms * 1e3, 1),
            "pct_hbm_peak": round(100 * value / world / peak, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": w.dtype, "data": "synthetic",
            "config": workload_config(w, args, n_arenas, world),
            "launch": {"how": ("one CUDA graph of the timed steps, replayed" if args.graph
                               else "one prepared gnmr_step call per step"),
                       "grid": grid_text(info)},
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                         "unit": "GB/s", "frac": round(achieved / peak, 4),
                         "traffic": traffic if args.shrink == 1 and args.group == "tensor" else None,
                         "traffic_unit": "bytes per launch (ncu dram__bytes_read+write)",
                         "algorithmic_bytes": w.grad_bytes,
                         "peak_source": f"{peak_kind} hbm_gbs", "kernel": f"gnmr_step_kernel<{w.dtype}>",
                         "kernel_ms_mean": round(kern_ms, 4),
                         "kernel_ms_median": round(statistics.median(per_ms), 4),
                         "kernel_ms_min": round(min(per_ms), 4)},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "e2e_staged": e2e_staged,
            "gpu_launches": launches,
            "clocks": clocks,
            "trigger_sparsity": sparsity,
        }
        if per_workload is not None:
            line["per_workload"] = per_workload
        print(json.dumps(line), flush=True)
    mon.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_actuator(args):
    """Fake-quant actuator over the saved input activations of every linear of
    the LLaMA-2-13B layout for one microbatch: unit b is a [tokens, in_features]
    bf16 block; 10 % of units take the recovery format (E4M3), the rest the
    low-cost one (E2M1).  Algorithmic bytes: one read and one write."""
    import torch
    import workloads
    from paper_2606_00539_gb300 import _native as N

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = workloads.make("llama2-13b", shrink=args.shrink)
    in_features = np.array([int(k) for k in _in_features(w)], np.int64)
    rows = np.full(w.num_units, args.tokens, np.int64)
    cols = in_features
    off = np.concatenate([[0], np.cumsum(rows * cols)[:-1]]).astype(np.int64)
    total = int((rows * cols).sum())
    acts = torch.empty(total, dtype=torch.bfloat16, device=dev)
    gen = torch.Generator(device=dev).manual_seed(0)
    for s0 in range(0, total, 1 << 28):
        n = min(1 << 28, total - s0)
        acts[s0:s0 + n] = torch.randn(n, generator=gen, device=dev).to(torch.bfloat16)
    out = torch.empty_like(acts)
    mask = (torch.rand(w.num_units, generator=gen, device=dev) < 0.1).to(torch.uint8)
    h = N.gnmr_actuator_create(off, rows, cols, N.GNMR_DTYPE_BF16, 0)
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    for _ in range(args.warmup):
        N.gnmr_actuator_apply(h, acts.data_ptr(), out.data_ptr(), total, mask.data_ptr(),
                              N.GNMR_FQ_E2M1, N.GNMR_FQ_E4M3, sp)
    stream.synchronize()
    sampler = ClockSampler(0)
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    wall0 = time.time()
    for i in range(args.steps):
        ev[i][0].record(stream)
        N.gnmr_actuator_apply(h, acts.data_ptr(), out.data_ptr(), total, mask.data_ptr(),
                              N.GNMR_FQ_E2M1, N.GNMR_FQ_E4M3, sp)
        ev[i][1].record(stream)
    stream.synchronize()
    wall1 = time.time()
    sampler.stop()
    N.gnmr_actuator_destroy(h)
    per_ms = [a.elapsed_time(b) for a, b in ev]
    ms = statistics.mean(per_ms)
    nbytes = 2 * total * 2
    peak, peak_kind = measured_peaks()
    gbs = nbytes / (ms / 1e3) / 1e9
    print(json.dumps({
        "metric": "GNMR recovery actuator: per-token fake quantization GB/s (read + write)",
        "value": round(gbs, 2), "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"llama2-13b input activations, {w.num_units} units x "
                               f"{args.tokens} tokens ({total} bf16 elements)",
                   "formats": "E2M1 low-cost, E4M3 recovery (10 % of units)",
                   "l2": "inputs larger than L2 (no flush)"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(gbs / peak, 4), "traffic": None,
                     "algorithmic_bytes": nbytes, "peak_source": f"{peak_kind} hbm_gbs",
                     "kernel": "fake_quant_kernel<bf16>", "kernel_ms_min": round(min(per_ms), 4)},
        "gpu_launches": args.steps, "clocks": sampler.summary(wall0, wall1),
    }), flush=True)


def run_static_norms(args):
    """gnmr_unit_norms_static on the workload's arena: per-unit norms with no
    allocation.  The layout is uploaded by the first (warm-up) call; the timed
    calls repeat it, as a training loop does.  Algorithmic bytes: the gradient
    read once."""
    import torch
    import workloads
    from paper_2606_00539_gb300 import _native as N

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = workloads.make(args.workload, shrink=args.shrink, group=args.group)
    filler = workloads.Filler(w, dev)
    arena = filler.new_arena()
    filler.fill(arena, w.steps // 2)
    out = torch.empty(w.num_units, dtype=torch.float64, device=dev)
    off = np.ascontiguousarray(w.offsets, np.int64)
    ln = np.ascontiguousarray(w.lengths, np.int64)
    if w.segment_unit is not None:
        raise SystemExit("static-norms times per-tensor units (--group tensor)")
    dt = N.GNMR_DTYPE_BF16 if w.dtype == "bf16" else N.GNMR_DTYPE_F32
    lib = N.load()
    stream = torch.cuda.Stream(dev)

    def call():
        st = lib.gnmr_unit_norms_static(arena.data_ptr(), arena.numel(), dt, w.num_units, off.ctypes.data,
                                        ln.ctypes.data, out.data_ptr(), stream.cuda_stream)
        if st != N.GNMR_OK:
            raise RuntimeError(f"gnmr_unit_norms_static: {N.status_string(st)}: {N.last_error(None)}")

    for _ in range(max(1, args.warmup)):
        call()
    stream.synchronize()
    sampler = ClockSampler(0)
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    wall0 = time.time()
    for i in range(args.steps):
        ev[i][0].record(stream)
        call()
        ev[i][1].record(stream)
    stream.synchronize()
    wall1 = time.time()
    sampler.stop()
    per_ms = [a.elapsed_time(b) for a, b in ev]
    ms = statistics.mean(per_ms)
    peak, peak_kind = measured_peaks()
    gbs = w.grad_bytes / (ms / 1e3) / 1e9
    print(json.dumps({
        "metric": "GNMR allocation-free per-unit norms GB/s (gradient read once)",
        "value": round(gbs, 2), "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": {"workload": f"{w.name} ({w.num_units} units, {w.grad_elems} {w.dtype} elements"
                               f"{'' if args.shrink == 1 else f', dims / {args.shrink}'})",
                   "l2": "inputs larger than L2 (no flush)" if w.grad_bytes > 2 * 129e6 else "inputs fit in L2 (hot)"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(gbs / peak, 4), "traffic": None, "algorithmic_bytes": w.grad_bytes,
                     "peak_source": f"{peak_kind} hbm_gbs", "kernel": f"static_norms_kernel<{w.dtype}>",
                     "kernel_ms_min": round(min(per_ms), 4)},
        "gpu_launches": args.steps, "clocks": sampler.summary(wall0, wall1),
    }), flush=True)


def _in_features(w):
    """Input width of every linear of a LLaMA layout (the saved activation of
    x @ W^T is [tokens, in_features])."""
    d = {"llama2-13b": (5120, 13824), "llama2-1.3b": (2048, 5504)}[w.name.split("/")[0]]
    out = []
    for k in w.kinds:
        name = k.split(".", 1)[1]
        out.append(d[1] if name == "down" else d[0])
    return out


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        run_reference(args)
    elif args.kernel == "actuator":
        run_actuator(args)
    elif args.kernel == "static-norms":
        run_static_norms(args)
    else:
        run_gnmr(args)


if __name__ == "__main__":
    main()

#!/usr/bin/env python
"""Benchmark of the BaryCache skipped-step forecast on GB300.

One step = one skipped diffusion step of the workload: the host weight solve (Diff Key memo,
Eqs. 8-12) plus the grouped forecast kernel over every cached layer (Eq. 13), issued through
the C ABI on a torch stream.  Inputs (the K history slots) are resident in HBM before the
timed region; they are far larger than L2 except for c2i-256, where L2 is flushed before
every step outside its events.  Steps alternate between the skipped steps that share one
history window, as in the equal-spaced schedule.

Prints one JSON line (rank 0).  Default workload: the video DiT (60 x [1, 118800, 3072] bf16,
K = 3; 131 GB of cache, 175 GB of HBM traffic per step).  Beside the headline the line
carries the roofline of the dominant kernel, the K sweep, the end-to-end leg with host
buffers, the oracle on the host cores, and the legs of the other rows (push, probe drift,
fused step, sampling loop, graph-captured loop, blockwise cache, other workloads).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload t2v|mmdit-t2i|t2i-1024|c2i-512|c2i-256] [--K 3] [--no-sweep]
                    [--no-e2e] [--no-cpu-baseline] [--no-clocks] [--no-extra]
                    [--e2e-steps S] [--e2e-chunk-layers C] [--probe-elems N]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "forecast HBM GB/s and % of GB300 peak; forecast elems/s; cache VRAM bytes"
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 126 * 2**20          # GB300 L2 (about 126 MiB usable)
NOMINAL_HBM_GBS = 8000.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="t2v")
    ap.add_argument("--K", type=int, default=None)
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip timing the workload's other history depths K")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--e2e-chunk-layers", type=int, default=6,
                    help="layers per pipelined chunk of the end-to-end leg")
    ap.add_argument("--e2e-host-cap-gb", type=float, default=48.0,
                    help="page-locked host memory for the e2e leg, shared by the node's ranks")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--probe-elems", type=int, default=None,
                    help="elements of the probe-drift leg (default: one layer)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the push and fused-step measurements")
    ap.add_argument("--warmup-min-s", type=float, default=None,
                    help="least wall time of every leg's warm-up (default 0.25 s; profiling "
                         "runs under ncu may shorten it)")
    ap.add_argument("--kernel", choices=["auto", "register", "pipeline"], default="auto",
                    help="pin the forecast kernel of the headline leg (default: the library's "
                         "choice)")
    return ap.parse_args()


# ----------------------------------------------------------------------------- helpers
def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            return float(json.load(fh)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_CODE_END = "// ------------------------------------------------------------------ launch plumbing"
# Warm-up lasts at least this long (wall time) as well as the requested number of steps:
# freeing a very large allocation (a previous leg's cache) costs HBM bandwidth for a while
# afterwards (about 70 ms after freeing 170 GB, at ~5.0 instead of ~7.1 TB/s), and a leg
# of short launches would otherwise time that transient.
MIN_WARMUP_S = 0.25


def _code_only(src: bytes) -> bytes:
    """Source text without comments or whitespace, so that editing a comment does not void
    a stored measurement."""
    import re
    text = src.decode()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    return re.sub(r"\s+", "", text).encode()


HOST_SIDE_START = "// ------------------------------------------------------------------ host side"


def kernel_source_hash(root: str = ROOT) -> str:
    """Hash of the forecast kernels' device code: bc_forecast_kernels.cuh up to its host
    launch plumbing (the tuning macros included), the kernel-visible part of bc_internal.h
    (layout, tiling, launch arguments; up to its host-side marker) and the pipeline
    primitives of bc_tma.cuh, comments and whitespace ignored.  A change there voids a stored
    ncu figure; host-side plumbing does not."""
    h = hashlib.sha256()
    csrc = os.path.join(root, "paper_2608_28670_gb300", "csrc")
    for name, marker in (("bc_forecast_kernels.cuh", KERNEL_CODE_END),
                         ("bc_internal.h", HOST_SIDE_START), ("bc_tma.cuh", None)):
        with open(os.path.join(csrc, name), "rb") as fh:
            text = fh.read()
        if marker is not None:
            text = text.split(marker.encode(), 1)[0]
        h.update(_code_only(text))
    return h.hexdigest()[:16]


def profiled_traffic(K: int, kernel: str, io: str = "bf16/bf16"):
    """DRAM bytes per output element of the forecast kernel (`kernel`: "pipeline" or
    "register") at history length K, from the committed ncu record, if one was taken with
    the current kernel source (else None).  The record comes from a small case (a few GB of
    cache); a launch moves the same bytes per element whatever its size, so the bench scales
    it by the elements of its own launch."""
    path = os.path.join(ROOT, "profiles", "forecast_kernel_traffic.json.txt")
    try:
        with open(path) as fh:
            rec = json.loads(fh.read().split("\n", 1)[1])  # first line is a comment
    except Exception:
        return None
    if rec.get("kernel_source_sha256_16") != kernel_source_hash():
        return None
    entry = rec.get("records", {}).get(f"K{K}/{kernel}/{io}")
    return entry.get("dram_bytes_per_output_element") if entry else None


class ClockSampler:
    """nvidia-smi samples every 100 ms, started before the warm-up (the tool takes a moment
    to start); stop(window) keeps the samples whose timestamps fall in the timed region."""

    def __init__(self, enabled: bool):
        self.proc = None
        self.path = None
        if not enabled:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")
        try:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
            local = int(os.environ.get("LOCAL_RANK", "0"))
            ids = [v for v in vis.split(",") if v] if vis else []
            idx = ids[local] if local < len(ids) else (ids[0] if ids else str(local))
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", idx, f"--query-gpu={q}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self, window=None):
        """Summary of the samples; `window` = (start, end) in time.time() seconds."""
        import datetime
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows, stamps = [], []
        with open(self.path) as fh:
            for line in fh:
                f = [x.strip() for x in line.split(",")]
                if len(f) >= 8:
                    try:
                        rows.append((float(f[1]), float(f[2]), float(f[3]), f[4:8]))
                        stamps.append(datetime.datetime.strptime(
                            f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp())
                    except ValueError:
                        pass
        os.unlink(self.path)
        if not rows:
            return None
        in_window = False
        if window is not None and len(stamps) == len(rows):
            kept = [r for r, t in zip(rows, stamps) if window[0] - 0.05 <= t <= window[1] + 0.05]
            if kept:
                rows, in_window = kept, True
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[3]) if v == "Active"})
        loaded = [r for r in rows if r[2] > 300.0] or rows
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows), "samples_under_load": len(loaded),
                "power_w_max": max(r[2] for r in rows),
                "samples_from": "timed region" if in_window else "warm-up and timed region"}


class nvtx_range:
    """NVTX range around a bench phase (shows up in Nsight timelines); no-op without CUDA."""

    def __init__(self, name: str):
        self.name = name

    def __enter__(self):
        try:
            import torch
            torch.cuda.nvtx.range_push(self.name)
            self.on = True
        except Exception:
            self.on = False
        return self

    def __exit__(self, *exc):
        if self.on:
            import torch
            torch.cuda.nvtx.range_pop()
        return False


# ----------------------------------------------------------------------------- ranks
def max_over_ranks(value: float, dist=None, device="cuda") -> float:
    """The slowest rank's value (time-like): all_reduce MAX, or the value itself at N = 1."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_rank: float, max_ms: float, world: int) -> float:
    """Whole-job GB/s of N replicas that each move `bytes_per_rank` in at most `max_ms`."""
    return bytes_per_rank * world / (max_ms * 1e-3) / 1e9


# ----------------------------------------------------------------------------- GPU arm
def window_targets(w, K):
    rep = w.representative(K)
    ts = [p.t for p in w.problems(K) if p.node_steps == rep.node_steps]
    return ts or [rep.t]


def warm_up(step, count, min_s=None):
    """Run `step(i)` at least `count` times and for at least `min_s` seconds of wall time
    (default MIN_WARMUP_S; synchronised); returns the number of steps run."""
    import torch
    min_s = MIN_WARMUP_S if min_s is None else min_s
    t0 = time.perf_counter()
    i = 0
    while i < count:
        step(i)
        i += 1
    torch.cuda.synchronize()
    while time.perf_counter() - t0 < min_s:
        for _ in range(4):
            step(i)
            i += 1
        torch.cuda.synchronize()
    return i


def time_forecast(run, steps, warmup, stream, dist=None):
    """Time `steps` skipped steps.  A workload whose step moves less than four L2s of data
    would be served from L2 back to back, so then L2 is flushed (a 512 MB write) before every
    step, outside that step's events, and the total is the sum of the steps."""
    import torch
    ts = window_targets(run.w, run.K)
    flush = None
    if run.algorithmic_bytes() < 4 * L2_BYTES:
        flush = torch.empty(512 * 2**20, dtype=torch.uint8, device="cuda")
    with nvtx_range("warmup"):
        warm_up(lambda i: run.forecast(ts[i % len(ts)]), warmup)
    if dist is not None:
        dist.barrier()
    st0 = run.stats()
    launches0 = st0["kernel_launches"]
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    host_s = []
    torch.cuda.synchronize()
    wall0 = time.time()
    with nvtx_range(f"timed {steps} skipped steps"):
        for i in range(steps):
            if flush is not None:
                flush.fill_(i & 0xFF)
            starts[i].record()
            h0 = time.perf_counter()
            run.forecast(ts[i % len(ts)])
            host_s.append(time.perf_counter() - h0)
            ends[i].record()
        torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    per_step = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_ms = sum(per_step) if flush is not None else starts[0].elapsed_time(ends[-1])
    time_forecast.l2 = ("flushed (512 MB write) before each step, outside its events"
                        if flush is not None else "inputs larger than L2 (no flush)")
    st1 = run.stats()
    launches = st1["kernel_launches"] - launches0
    time_forecast.window = (wall0, time.time())
    time_forecast.host_us = 1e6 * statistics.median(host_s)
    time_forecast.pipeline = st1["pipeline_launches"] - st0["pipeline_launches"]
    return total_ms, per_step, launches


def run_ours(args):
    global MIN_WARMUP_S
    if args.warmup_min_s is not None:
        MIN_WARMUP_S = max(0.0, args.warmup_min_s)
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    from paper_2608_28670_gb300.configs import WORKLOADS, T2V_HBM_BUDGET
    from paper_2608_28670_gb300.runner import WorkloadRun
    import __graft_entry__

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as tdist
        torch.cuda.set_device(local)
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local))
        dist = tdist
    else:
        torch.cuda.set_device(0)
    __graft_entry__.build_libraries()   # no-op when the libraries are current
    w = WORKLOADS[args.workload]
    K = args.K or w.K
    budget = T2V_HBM_BUDGET if w.name == "t2v" else None
    stream = torch.cuda.current_stream().cuda_stream

    run = WorkloadRun(w, K=K, budget_bytes=budget, stream=stream)
    kernel_choice = {"auto": bc.KERNEL_AUTO, "register": bc.KERNEL_REGISTER,
                     "pipeline": bc.KERNEL_PIPELINE}[args.kernel]
    bc.bc_cache_set_kernel(run.h, kernel_choice)
    try:
        torch.cuda.synchronize()
        clocks = ClockSampler(not args.no_clocks)
        total_ms, per_step, launches = time_forecast(run, args.steps, args.warmup, stream, dist)
        clk = clocks.stop(time_forecast.window)
        ms = max_over_ranks(total_ms / args.steps, dist)
        alg = run.algorithmic_bytes()
        value = job_throughput(alg, ms, world)
        elems = run.w.layer_numel * run.n_feat + (run.numels[-1] if run.euler else 0)
        launches_per_step = launches / args.steps
        kernel_ms = statistics.mean(per_step) / max(launches_per_step, 1)
        per_launch_bytes = alg / max(launches_per_step, 1)
        peak, peak_kind = measured_peak()
        achieved = per_launch_bytes / (kernel_ms * 1e-3) / 1e9
        kernel_kind = "pipeline" if time_forecast.pipeline == launches else "register"
        io = "bf16/bf16" if w.dtype == bc.DTYPE_BF16 else "f32/f32"
        traffic_per_elem = None if w.euler_shape else profiled_traffic(K, kernel_kind, io)
        per_launch_elems = elems / max(launches_per_step, 1)
        result = {
            "metric": METRIC, "value": round(value, 1), "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {
                "workload": w.name,
                "layers": f"{w.n_layers}x{list(w.layer_shape)}"
                          + (f" + euler {list(w.euler_shape)}" if w.euler_shape else ""),
                "storage_dtype": "bf16" if w.dtype == bc.DTYPE_BF16 else "f32",
                "K": K, "forecast_calls_per_step": run.calls,
                "layers_per_call": run.window,
                "weights": "paper Eqs. 8-12, delta_H table, lambda 0, C 10, eta 1e-12",
                "targets": window_targets(w, K), "nodes": list(run.problem.nodes),
                "l2": time_forecast.l2,
                "kernel_choice": args.kernel,
                "warmup_s_min": MIN_WARMUP_S,
                "parallelism": f"replicas x{world}",
            },
            "pct_of_measured_peak": round(100 * value / world / peak, 2),
            "pct_of_nominal_8tbs": round(100 * value / world / NOMINAL_HBM_GBS, 2),
            "elems_per_s": round(elems * world / (ms * 1e-3), 1),
            "per_skipped_step_ms": round(ms, 4),
            "cache_bytes": bc.bc_cache_bytes(run.h),
            "algorithmic_bytes_per_step": alg,
            "roofline": {
                "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                "unit": "GB/s", "frac": round(achieved / peak, 4), "peak_kind": peak_kind,
                "nominal_peak": NOMINAL_HBM_GBS,
                "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                "traffic": (round(traffic_per_elem * per_launch_elems)
                            if traffic_per_elem else None),
                "traffic_source": ("ncu dram__bytes_read.sum + dram__bytes_write.sum per output "
                                   "element on t2i-1024-shaped launches (profiles/"
                                   "forecast_kernel_traffic.json.txt), times this launch's "
                                   "output elements" if traffic_per_elem else
                                   "no ncu record for this kernel source, K and kernel"),
                "kernel": ("bc::forecast_tma_kernel (TMA pipeline)"
                           if kernel_kind == "pipeline" else "bc::forecast_kernel"),
                "avg_launch_ms": round(kernel_ms, 4),
                "algorithmic_bytes_per_launch": per_launch_bytes,
            },
            "gpu_launches": launches,
            "step_ms": {"min": round(min(per_step), 4),
                        "median": round(statistics.median(per_step), 4),
                        "max": round(max(per_step), 4), "first": round(per_step[0], 4)},
            "host_call_us": round(time_forecast.host_us, 1),
        }
        if clk:
            result["clocks"] = clk
        if not args.no_sweep and w.K_sweep:
            sweep = {}
            run.close()
            run = None
            torch.cuda.empty_cache()
            for k in w.K_sweep:
                r = WorkloadRun(w, K=k, budget_bytes=budget, stream=stream)
                bc.bc_cache_set_kernel(r.h, kernel_choice)
                try:
                    tm, ps, ln = time_forecast(r, args.steps, args.warmup, stream, dist)
                    a = r.algorithmic_bytes()
                    m = tm / args.steps
                    kk = "pipeline" if time_forecast.pipeline == ln else "register"
                    per = profiled_traffic(k, kk, io)
                    lpl = ln / args.steps                       # launches per step
                    gbs = a / (m * 1e-3) / 1e9
                    sweep[f"K{k}"] = {"GB/s": round(gbs, 1), "ms": round(m, 4),
                                      "frac": round(gbs / peak, 4),
                                      "frac_of_nominal": round(gbs / NOMINAL_HBM_GBS, 4),
                                      "cache_bytes": bc.bc_cache_bytes(r.h),
                                      "calls_per_step": r.calls, "layers_per_call": r.window,
                                      "launches": ln, "kernel": kk,
                                      "algorithmic_bytes_per_launch": a / lpl,
                                      "traffic": (round(per * r.w.layer_numel * r.n_feat / lpl)
                                                  if per else None)}
                finally:
                    r.close()
                    torch.cuda.empty_cache()
            result["sweep"] = sweep
            run = WorkloadRun(w, K=K, budget_bytes=budget, stream=stream)
        if not args.no_e2e:      # before the CPU leg, which loads the host memory system
            with nvtx_range("e2e"):
                result["e2e"] = e2e(run, args.e2e_steps, world, dist,
                                    chunk_layers=args.e2e_chunk_layers,
                                    host_cap_bytes=args.e2e_host_cap_gb * 1e9)
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            with nvtx_range("cpu_baseline"):
                result["cpu_baseline"] = cpu_baseline_from_device(run, args.cpu_seconds)
        if not args.no_extra:
            with nvtx_range("probe_drift"):
                result["probe_drift"] = time_probe(run, args.steps, args.probe_elems)
            with nvtx_range("push"):
                result["push"] = time_push(run, args.steps)
    finally:
        if run is not None:
            run.close()
    cpu_legs = rank == 0 and world == 1 and not args.no_cpu_baseline
    if not args.no_extra and w.name != "mmdit-t2i":
        torch.cuda.empty_cache()
        with nvtx_range("fused_step"):
            result["fused_step"] = time_fused(args, stream, dist, cpu=cpu_legs)
    if not args.no_extra:
        torch.cuda.empty_cache()
        with nvtx_range("sampling_loop"):
            result["sampling_loop"] = time_sampling_loop(stream)
        torch.cuda.empty_cache()
        with nvtx_range("graph_loop"):
            result["graph_loop"] = time_graph_loop(stream)
        with nvtx_range("blockwise"):
            result["blockwise"] = time_blockwise(stream, args.steps)
        torch.cuda.empty_cache()
        with nvtx_range("other_workloads"):
            result["other_workloads"] = time_other_workloads(stream, args.steps, cpu=cpu_legs)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(result), flush=True)


def _continuation(run, i):
    """(time of the i-th next full step, the skipped step after it) continuing the window's
    spacing."""
    p = run.problem
    nodes = p.nodes
    step = (nodes[0] - nodes[1]) if len(nodes) > 1 else 2.0 * (p.t - nodes[0])
    off = p.t - nodes[0]
    t_full = nodes[0] + (i + 1) * step
    return t_full, t_full + off


def time_push(run, steps):
    """Row a2, copy path: bc_cache_push of one full slot (every layer) from device buffers
    (the forecast outputs stand in for a full step's features); 2 bytes of HBM traffic per
    byte of slot.  Only when the outputs cover every layer."""
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    if run.window < run.n_feat or run.euler:
        return None
    import numpy as np
    ptrs = np.array([o.data_ptr() for o in run.outs], dtype=np.uint64)
    slot = sum(n * run.w.elem_bytes for n in run.numels)
    counter = [100]

    def push(_i=0):
        bc.bc_cache_push(run.h, ptrs, _continuation(run, counter[0])[0], run.stream)
        counter[0] += 1

    def timed(kernel):
        bc.bc_cache_set_kernel(run.h, kernel)
        warm_up(push, 2)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record()
        for i in range(steps):
            push()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / steps

    gbs = lambda ms: round(2 * slot / (ms * 1e-3) / 1e9, 1)
    by_kernel = {"register": gbs(timed(bc.KERNEL_REGISTER)),
                 "pipeline": gbs(timed(bc.KERNEL_PIPELINE))}
    ms = timed(bc.KERNEL_AUTO)
    bc.bc_cache_check(run.h)
    return {"GB/s": gbs(ms), "ms": round(ms, 4), "GB/s_by_kernel": by_kernel,
            "bytes_per_push": 2 * slot, "pushes": steps,
            "what": "grouped byte-exact copy of one slot (read + write)"}


def time_probe(run, steps, probe_elems=None):
    """Row f3: the probe drift of the adaptive schedule over one cached layer (newest vs the
    previous node's copy of layer 0): 2 x numel x b bytes, two launches per call.
    `probe_elems` probes that many elements from the start of the two slots instead (a
    flat view across layers; at most one slot)."""
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    if len(run.problem.nodes) < 2:
        return None
    n = run.numels[0]
    if probe_elems:
        n = min(int(probe_elems), bc.bc_cache_layout(run.h)[-1] // run.w.elem_bytes)
    cur = bc.bc_cache_slot_ptrs(run.h, 0, len(run.numels))[0]
    prev = bc.bc_cache_slot_ptrs(run.h, 1, len(run.numels))[0]
    out = torch.empty(3, dtype=torch.float64, device="cuda")
    warm_up(lambda i: bc.bc_probe_drift(run.h, cur, prev, n, run.w.dtype, out.data_ptr(),
                                        run.stream), 3)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record()
    for _ in range(steps):
        bc.bc_probe_drift(run.h, cur, prev, n, run.w.dtype, out.data_ptr(), run.stream)
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / steps
    nbytes = 2 * n * run.w.elem_bytes
    # a realistic adaptive-schedule probe is a few MB and latency-bound: the device time of
    # one call on a DiT-XL/2 256 px block output's worth of elements (589,824 of the cache
    # dtype), 100 calls replayed from a CUDA graph so that the host's per-call cost is not
    # what is timed (the probe stays in L2 between calls)
    small_n = min(589824, n)
    g = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
            for _ in range(100):
                bc.bc_probe_drift(run.h, cur, prev, small_n, run.w.dtype, out.data_ptr(),
                                  side.cuda_stream)
    g.replay()
    torch.cuda.synchronize()
    a.record()
    g.replay()
    b.record()
    torch.cuda.synchronize()
    small_us = 1e3 * a.elapsed_time(b) / 100
    return {"GB/s": round(nbytes / (ms * 1e-3) / 1e9, 1), "ms": round(ms, 4),
            "elements": n, "bytes_per_call": nbytes, "drift": round(float(out[2].item()), 6),
            "small_probe_us": round(small_us, 2), "small_probe_elements": small_n,
            "what": "bc_probe_drift over layer 0 (newest vs previous node)" if not probe_elems
                    else "bc_probe_drift over the first elements of the two newest slots"}


def time_sampling_loop(stream):
    """Row f1: a whole 28-step flow sampler on the MMDiT workload (57 block outputs + the
    velocity), equal-spaced schedule with N = 3 and K = 3.  Full steps: a stand-in model
    (the seeded generator) writes every layer's new feature straight into the next cache slot,
    the slot is committed, and the Euler step uses the written velocity; skipped steps: one
    fused forecast + Euler launch over every layer.  Reports the device time of both kinds of
    step; the stand-in's time says nothing about a real DiT."""
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    from paper_2608_28670_gb300 import synth
    from paper_2608_28670_gb300.configs import WORKLOADS
    from paper_2608_28670_gb300.runner import device_view
    w = WORKLOADS["mmdit-t2i"]
    K = w.K
    ts = w.times() + [0.0]
    sched = bc.bc_schedule_equal(w.steps, w.interval, K)
    numels = w.numels
    L = len(numels)
    h = bc.bc_cache_create(numels, K, w.dtype)
    try:
        tdt = torch.bfloat16
        outs = [torch.empty(w.layer_numel, dtype=tdt, device="cuda") for _ in range(w.n_layers)]
        x = torch.zeros(numels[-1], dtype=torch.float32, device="cuda")
        full_ms, skip_ms = [], []
        for rep in range(2):                   # the first pass warms up
            bc.bc_cache_reset(h)
            full_ms, skip_ms = [], []
            for i in range(w.steps):
                t, dt = ts[i], ts[i + 1] - ts[i]
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record()
                if sched[i]:
                    slots = bc.bc_cache_next_slot_ptrs(h, L)
                    for l, n in enumerate(numels):
                        synth.fill_device(slots[l], w.dtype, n, seed=2026, tensor_id=l,
                                          step_id=i, tau=t, degree=w.degree,
                                          noise_std=w.noise_std, stream=stream)
                    bc.bc_cache_commit(h, t)
                    v = device_view(slots[-1], numels[-1], w.dtype).view(tdt)
                    x.add_(v.float(), alpha=dt)
                else:
                    bc.bc_forecast_step(h, t, dt, [o.data_ptr() for o in outs] + [None],
                                        w.dtype, L - 1, x.data_ptr(), bc.DTYPE_F32, stream)
                b.record()
                (full_ms if sched[i] else skip_ms).append((a, b))
            torch.cuda.synchronize()
        f = [a.elapsed_time(b) for a, b in full_ms]
        sk = [a.elapsed_time(b) for a, b in skip_ms]
        st = bc.bc_cache_stats(h)
        return {"workload": "mmdit-t2i", "steps": w.steps, "full_steps": len(f),
                "skipped_steps": len(sk), "skipped_step_ms": round(statistics.mean(sk), 4),
                "skipped_total_ms": round(sum(sk), 3),
                "standin_full_step_ms": round(statistics.mean(f), 4),
                "forecast_GB/s": round(w.forecast_bytes(K, x_elem_bytes=4) /
                                       (statistics.mean(sk) * 1e-3) / 1e9, 1),
                "memo_hits": st["memo_hits"], "memo_misses": st["memo_misses"],
                "what": "28-step flow sampler, equal-spaced N=3, K=3; full steps = seeded "
                        "stand-in writing the next slot in place"}
    finally:
        bc.bc_cache_destroy(h)


def time_graph_loop(stream):
    """Row f1 on the latency-bound DiT-XL/2 256 px workload, eager and as one CUDA graph:
    a 50-step DDIM sampler (equal-spaced N = 3, K = 3) over the cached block output
    [2, 256, 1152] fp32 plus the eps prediction [2, 4, 32, 32].  Full steps: the stand-in
    (seeded generator) writes both tensors into the next slot and x takes the DDIM step
    from the written eps; skipped steps: one fused forecast + DDIM launch.  The whole loop is
    captured once and replayed; each replay repeats the captured device work (same slots
    and weights).  Per-step kernels are a few microseconds here, so the eager loop is bound
    by the host's per-call cost and the replay shows what the device needs."""
    import numpy as np
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    from paper_2608_28670_gb300 import synth
    from paper_2608_28670_gb300.runner import device_view
    steps, interval, K = 50, 3, 3
    numels = [2 * 256 * 1152, 2 * 4 * 32 * 32]
    ts = [980.0 - 20.0 * i for i in range(steps)]
    ab = np.cumprod(1.0 - np.linspace(1e-4, 0.02, 1000))
    coef = [bc.bc_ddim_coefficients(ab[int(t)], ab[int(t) - 20] if t >= 20 else 1.0, 0.0)
            for t in ts]
    sched = bc.bc_schedule_equal(steps, interval, K)
    h = bc.bc_cache_create(numels, K, bc.DTYPE_F32)
    side = torch.cuda.Stream()
    try:
        out = torch.empty(numels[0], device="cuda")
        x0 = torch.linspace(-1.0, 1.0, numels[1], device="cuda")
        x = x0.clone()

        def loop(s):
            for i in range(steps):
                a, b, _ = coef[i]
                if sched[i]:
                    slots = bc.bc_cache_next_slot_ptrs(h, 2)
                    for l, n in enumerate(numels):
                        synth.fill_device(slots[l], bc.DTYPE_F32, n, seed=2026, tensor_id=l,
                                          step_id=i, tau=ts[i] / 1000.0, degree=2,
                                          noise_std=1e-3, stream=s)
                    bc.bc_cache_commit(h, ts[i])
                    x.mul_(a).add_(device_view(slots[1], numels[1], bc.DTYPE_F32), alpha=b)
                else:
                    bc.bc_forecast_update(h, ts[i], a, b, 0.0, [out.data_ptr(), None],
                                          bc.DTYPE_F32, 1, x.data_ptr(), bc.DTYPE_F32, None, s)

        def timed(fn, reps):
            ms = []
            for _ in range(reps):
                x.copy_(x0)
                bc.bc_cache_reset(h)
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                fn()
                b.record()
                torch.cuda.synchronize()
                ms.append(a.elapsed_time(b))
            return statistics.median(ms)

        with torch.cuda.stream(side):
            sid = side.cuda_stream
            st0 = bc.bc_cache_stats(h)
            eager_ms = timed(lambda: loop(sid), 5)
            x_eager = x.clone()
            st1 = bc.bc_cache_stats(h)
        launches = (st1["kernel_launches"] - st0["kernel_launches"]) // 5
        g = torch.cuda.CUDAGraph()
        bc.bc_cache_reset(h)
        x.copy_(x0)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            loop(torch.cuda.current_stream().cuda_stream)
        graph_ms = timed(g.replay, 20)
        same = bool(torch.equal(x, x_eager))
        n_skip = steps - sum(sched)
        return {"workload": "c2i-256 + eps [2, 4, 32, 32], DDIM-50, N=3, K=3",
                "steps": steps, "full_steps": sum(sched), "skipped_steps": n_skip,
                "eager_loop_ms": round(eager_ms, 3), "graph_loop_ms": round(graph_ms, 3),
                "eager_us_per_step": round(1e3 * eager_ms / steps, 2),
                "graph_us_per_step": round(1e3 * graph_ms / steps, 2),
                "library_launches_per_loop": launches,
                "graph_equals_eager": same,
                "what": "whole sampling loop captured once into a CUDA graph and replayed"}
    finally:
        bc.bc_cache_destroy(h)


def time_blockwise(stream, steps):
    """Row f2: a many-tensor (blockwise) cache -- 4096 tensors of 65,536 bf16 elements, K = 3
    (1.6 GB of cache) -- forecast through per-layer output pointers (one launch reading its
    layer table from the handle's device copy, uploaded once for these outputs) and through
    one flat slot-shaped output (one launch); its full-step push from per-tensor sources and
    from one slot-shaped buffer (bc_cache_push_flat)."""
    import numpy as np
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    from paper_2608_28670_gb300 import synth
    n_t, n = 4096, 65536
    numels = [n] * n_t
    h = bc.bc_cache_create(numels, 3, bc.DTYPE_BF16)
    try:
        for j, t in enumerate((0.9, 0.85, 0.8)):
            slots = bc.bc_cache_next_slot_ptrs(h, n_t)
            offs = bc.bc_cache_layout(h, n_t)
            synth.fill_device(slots[0], bc.DTYPE_BF16, offs[-1] // 2, seed=7, tensor_id=0,
                              step_id=j, tau=t, degree=2, noise_std=1e-2, stream=stream)
            bc.bc_cache_commit(h, t)
        offs = bc.bc_cache_layout(h, n_t)
        flat = torch.empty(offs[-1] // 2, dtype=torch.bfloat16, device="cuda")
        per = np.array([flat.data_ptr() + offs[l] for l in range(n_t)], dtype=np.uint64)
        alg = (3 * 2 + 2) * n * n_t

        def timed(fn):
            warm_up(lambda i: fn(), 3)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            l0 = bc.bc_cache_stats(h)["kernel_launches"]
            a.record()
            for _ in range(steps):
                fn()
            b.record()
            torch.cuda.synchronize()
            timed.launches = (bc.bc_cache_stats(h)["kernel_launches"] - l0) / steps
            return a.elapsed_time(b) / steps
        by_kernel = {}
        for name, kern in (("register", bc.KERNEL_REGISTER), ("pipeline", bc.KERNEL_PIPELINE),
                           ("auto", bc.KERNEL_AUTO)):
            bc.bc_cache_set_kernel(h, kern)
            by_kernel[name] = round(alg / (timed(
                lambda: bc.bc_forecast(h, 0.75, per, bc.DTYPE_BF16, stream)) * 1e-3) / 1e9, 1)
        ms_layers = timed(lambda: bc.bc_forecast(h, 0.75, per, bc.DTYPE_BF16, stream))
        per_layer_launches = timed.launches
        st = bc.bc_cache_stats(h)
        ms_flat = timed(lambda: bc.bc_forecast_flat(h, 0.75, flat.data_ptr(), stream))
        flat_launches = timed.launches
        # the full step of a blockwise cache: push every tensor (from the forecast's buffers)
        push_t = [0.7 - 1e-4 * i for i in range(100000)]
        k = [0]

        def push():
            bc.bc_cache_push(h, per, push_t[k[0]], stream)
            k[0] += 1
        push_bytes = 2 * 2 * n * n_t
        push_by_kernel = {}
        for name, kern in (("register", bc.KERNEL_REGISTER), ("pipeline", bc.KERNEL_PIPELINE)):
            bc.bc_cache_set_kernel(h, kern)
            push_by_kernel[name] = round(push_bytes / (timed(push) * 1e-3) / 1e9, 1)
        bc.bc_cache_set_kernel(h, bc.KERNEL_AUTO)
        ms_push = timed(push)
        push_launches = timed.launches
        uploads = bc.bc_cache_stats(h)["table_uploads"] - st["table_uploads"]

        def push_flat():            # the same step from one slot-shaped buffer
            bc.bc_cache_push_flat(h, flat.data_ptr(), push_t[k[0]], stream)
            k[0] += 1
        ms_push_flat = timed(push_flat)
        push_flat_launches = timed.launches
        return {"tensors": n_t, "elements_per_tensor": n,
                "per_layer": {"GB/s": round(alg / (ms_layers * 1e-3) / 1e9, 1),
                              "ms": round(ms_layers, 4),
                              "launches_per_call": per_layer_launches,
                              "table_uploads": st["table_uploads"],
                              "GB/s_by_kernel": by_kernel},
                "flat": {"GB/s": round(alg / (ms_flat * 1e-3) / 1e9, 1), "ms": round(ms_flat, 4),
                         "launches_per_call": flat_launches},
                "push": {"GB/s": round(push_bytes / (ms_push * 1e-3) / 1e9, 1),
                         "ms": round(ms_push, 4), "launches_per_call": push_launches,
                         "GB/s_by_kernel": push_by_kernel,
                         "bytes_per_push": push_bytes,
                         "table_uploads": uploads},
                "push_flat": {"GB/s": round(push_bytes / (ms_push_flat * 1e-3) / 1e9, 1),
                              "ms": round(ms_push_flat, 4),
                              "launches_per_call": push_flat_launches}}
    finally:
        bc.bc_cache_destroy(h)


def time_other_workloads(stream, steps, cpu=False):
    """The remaining workloads: c2i-256 (9.4 MB per forecast, L2-resident, so L2 is flushed
    by writing 512 MB before every timed launch, outside its event pair; the flush keeps the
    device busy while the host enqueues the forecast; `us_after_clean_flush` adds a 512 MB
    read after the write, so that no dirty line is left for the forecast to write back),
    c2i-512 (K = 4, 2.6 GB) and t2i-1024
    (K = 3, 4.2 GB), whose inputs exceed L2: `steps` forecasts back to back between one event
    pair, as in the headline measurement.  `idle_start_us` is one call on an idle device
    (host call to completion: memo lookup, table build and launch latency included).  With
    `cpu`, each entry also carries the oracle over the whole workload (cpu_baseline_full)."""
    import torch
    from paper_2608_28670_gb300.configs import WORKLOADS
    from paper_2608_28670_gb300.runner import WorkloadRun
    flush = torch.empty(512 * 2**20, dtype=torch.uint8, device="cuda")
    clean = torch.zeros(128 * 2**20, dtype=torch.int32, device="cuda")   # 512 MB, read only
    out = {}

    def pair():
        return torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    for name in ("c2i-256", "c2i-512", "t2i-1024"):
        w = WORKLOADS[name]
        r = WorkloadRun(w, stream=stream)
        try:
            warm_up(lambda i: r.forecast(), 3)
            p0 = r.stats()["pipeline_launches"]
            warm_us = clean_us = floor_us = None
            if name == "c2i-256":
                ms = []
                for i in range(steps):
                    flush.fill_(i & 0xFF)
                    a, b = pair()
                    a.record()
                    r.forecast()
                    b.record()
                    torch.cuda.synchronize()
                    ms.append(a.elapsed_time(b))
                m = statistics.median(ms)
                # the same after a flush that leaves L2 clean: the write, then a 512 MB read
                # (both outside the events), so that the forecast reads its history from HBM
                # without also writing back the flush's dirty lines it evicts
                ms_clean = []
                for i in range(steps):
                    flush.fill_(i & 0xFF)
                    clean.sum()
                    a, b = pair()
                    a.record()
                    r.forecast()
                    b.record()
                    torch.cuda.synchronize()
                    ms_clean.append(a.elapsed_time(b))
                clean_us = round(1e3 * statistics.median(ms_clean), 1)
                # the floor of that measurement: a one-element fill, timed the same way
                tiny = torch.zeros(1, dtype=torch.int32, device="cuda")
                ms_floor = []
                for i in range(steps):
                    flush.fill_(i & 0xFF)
                    clean.sum()
                    a, b = pair()
                    a.record()
                    tiny.fill_(i)
                    b.record()
                    torch.cuda.synchronize()
                    ms_floor.append(a.elapsed_time(b))
                floor_us = round(1e3 * statistics.median(ms_floor), 1)
                # beside it: launches back to back with the 9.4 MB resident in L2, replayed
                # from a CUDA graph so that the host's per-call cost is not what is timed
                g = torch.cuda.CUDAGraph()
                side = torch.cuda.Stream()
                with torch.cuda.stream(side):
                    r.stream = side.cuda_stream
                    with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
                        for _ in range(100):
                            r.forecast()
                    r.stream = stream
                g.replay()
                torch.cuda.synchronize()
                a, b = pair()
                a.record()
                g.replay()
                b.record()
                torch.cuda.synchronize()
                warm_us = round(1e3 * a.elapsed_time(b) / 100, 2)
            else:
                a, b = pair()
                a.record()
                for _ in range(steps):
                    r.forecast()
                b.record()
                torch.cuda.synchronize()
                m = a.elapsed_time(b) / steps
            pipe = r.stats()["pipeline_launches"] - p0
            idle = []
            for _ in range(5):
                torch.cuda.synchronize()
                a, b = pair()
                a.record()
                r.forecast()
                b.record()
                torch.cuda.synchronize()
                idle.append(a.elapsed_time(b))
            gbs = r.algorithmic_bytes() / (m * 1e-3) / 1e9
            out[name] = {"GB/s": round(gbs, 1), "us": round(1e3 * m, 1),
                         "bytes": r.algorithmic_bytes(),
                         "elems_per_s": round(r.w.layer_numel * r.n_feat / (m * 1e-3), 1),
                         "idle_start_us": round(1e3 * statistics.median(idle), 1),
                         "l2_warm_back_to_back_us": warm_us,
                         "us_after_clean_flush": clean_us,
                         "one_element_kernel_us_after_clean_flush": floor_us,
                         "K": r.K, "pipeline_kernel": pipe > 0,
                         "cache_bytes": bc_cache_bytes(r),
                         "l2": "flushed before each launch" if name == "c2i-256"
                               else "inputs larger than L2, launches back to back"}
            if cpu:
                out[name]["cpu_baseline"] = cpu_baseline_full(r)
        finally:
            r.close()
    return out


def bc_cache_bytes(run):
    from paper_2608_28670_gb300 import barycache as bc
    return bc.bc_cache_bytes(run.h)


def time_fused(args, stream, dist, cpu=False):
    """Row a4: the fused forecast + Euler step on the MMDiT workload (57 block outputs plus
    the velocity [1, 16, 128, 128], one launch per step); with `cpu`, the oracle over the
    whole step beside it."""
    from paper_2608_28670_gb300.configs import WORKLOADS
    from paper_2608_28670_gb300.runner import WorkloadRun
    r = WorkloadRun(WORKLOADS["mmdit-t2i"], stream=stream)
    try:
        tm, ps, ln = time_forecast(r, args.steps, args.warmup, stream, dist)
        ms = tm / args.steps
        a = r.algorithmic_bytes()
        res = {"workload": "mmdit-t2i", "GB/s": round(a / (ms * 1e-3) / 1e9, 1),
               "ms": round(ms, 4), "algorithmic_bytes_per_step": a, "launches": ln,
               "elems_per_s": round(sum(r.numels) / (ms * 1e-3), 1),
               "cache_bytes": bc_cache_bytes(r), "steps": args.steps}
        if cpu:
            res["cpu_baseline"] = cpu_baseline_full(r)
        return res
    finally:
        r.close()


def pinned_host_buffer(nbytes):
    """Page-locked host memory of exactly `nbytes`: cudaHostAlloc through the CUDA runtime
    that torch loaded, else cudaHostRegister of a numpy buffer.  Returns (uint8 array,
    release function, description)."""
    import ctypes
    import glob
    import numpy as np
    import torch
    rt = None
    cands = ["libcudart.so.13"] + sorted(glob.glob(os.path.join(
        os.path.dirname(torch.__file__), "..", "nvidia", "*", "lib", "libcudart.so*")))
    for c in cands:
        try:
            rt = ctypes.CDLL(c)
            break
        except OSError:
            continue
    if rt is not None:
        ptr = ctypes.c_void_p()
        rt.cudaHostAlloc.argtypes = [ctypes.POINTER(ctypes.c_void_p), ctypes.c_size_t,
                                     ctypes.c_uint]
        rt.cudaFreeHost.argtypes = [ctypes.c_void_p]
        if rt.cudaHostAlloc(ctypes.byref(ptr), nbytes, 0) == 0 and ptr.value:
            arr = np.ctypeslib.as_array((ctypes.c_uint8 * nbytes).from_address(ptr.value))
            return arr, (lambda: rt.cudaFreeHost(ptr)), "cudaHostAlloc"
    arr = np.empty(nbytes, dtype=np.uint8)
    cudart = torch.cuda.cudart()
    if int(cudart.cudaHostRegister(arr.ctypes.data, nbytes, 0)) != 0:
        return None, None, f"no page-locked host buffer of {nbytes} bytes"
    return arr, (lambda: cudart.cudaHostUnregister(arr.ctypes.data)), "cudaHostRegister"


def link_probe(host, nbytes, chunks=10):
    """Sustained copy-engine throughput of this machine's host link over the whole of the e2e
    leg's pinned buffer (bursts of a few GB run faster than the link sustains): H2D of every
    chunk, D2H of every chunk, and both directions at once on two streams (chunk c in while
    chunk c + chunks/2 goes out), GB/s, the best of two passes after one untimed pass.  Runs
    before the buffer is filled (its D2H writes the buffer)."""
    import torch
    n = int(nbytes) // chunks // 4096 * 4096
    if n < 4096:
        return None
    hv = torch.from_numpy(host)
    dev_a = torch.empty(n, dtype=torch.uint8, device="cuda")
    dev_b = torch.zeros(n, dtype=torch.uint8, device="cuda")
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    part = [slice(c * n, (c + 1) * n) for c in range(chunks)]

    def h2d():
        for c in range(chunks):
            dev_a.copy_(hv[part[c]], non_blocking=True)

    def d2h():
        for c in range(chunks):
            hv[part[c]].copy_(dev_b, non_blocking=True)

    def both():
        for c in range(chunks):
            with torch.cuda.stream(s1):
                dev_a.copy_(hv[part[c]], non_blocking=True)
            with torch.cuda.stream(s2):
                hv[part[(c + chunks // 2) % chunks]].copy_(dev_b, non_blocking=True)
        torch.cuda.current_stream().wait_stream(s1)
        torch.cuda.current_stream().wait_stream(s2)

    def rate(fn, moved):
        fn()
        best = None
        for _ in range(2):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            g = moved / (time.perf_counter() - t0) / 1e9
            best = g if best is None else max(best, g)
        return round(best, 1)

    out = {"bytes_each_way": n * chunks, "h2d_GB/s": rate(h2d, n * chunks),
           "d2h_GB/s": rate(d2h, n * chunks), "both_GB/s": rate(both, 2 * n * chunks)}
    del dev_a, dev_b
    return out


def e2e(run, steps, world, dist, chunk_layers=6, host_cap_bytes=48 * 10**9):
    """Same metric through the public API with host buffers.  Per step: the new full-step
    features (one slot, every layer) are copied from pinned host memory into the next cache
    slot and committed (zero-copy push, Eq. 6), the following skipped step is forecast, and
    the forecast is read back into pinned host memory.  One pinned host buffer of one slot
    serves both directions (the read-back of step i is the input of step i + 1).

    The transfers are pipelined by chunks of layers on three streams: host->device copies of
    chunk c, the forecast of chunk c (bc_forecast with the other outputs NULL) once they have
    landed, and the device->host copy of its output; the next step's copy into chunk c waits
    for this step's read-back of chunk c (which itself follows the forecast that read the slot
    being overwritten)."""
    import numpy as np
    import torch
    from paper_2608_28670_gb300 import barycache as bc
    from paper_2608_28670_gb300.runner import device_view

    if run.euler:
        return {"unavailable": "e2e is measured on workloads without the Euler layer"}
    eb = run.w.elem_bytes
    ob = 2 if run.out_dtype == bc.DTYPE_BF16 else 4
    if ob != eb:
        return {"unavailable": "e2e reuses the input buffer for the output: dtypes differ"}
    sizes = [n * eb for n in run.numels]
    total = int(sum(sizes))
    # Page-locked host memory per rank is capped (48 GB shared by the ranks of one node):
    # when a slot does not fit, layers cycle through a ring of host buffers, so every step
    # still moves a whole slot each way over the host link.
    cap = int(host_cap_bytes) // max(world, 1)
    if total <= cap:
        offs = np.cumsum([0] + sizes)
        host_bytes = total
    else:
        per = max(sizes)
        ring = max(1, cap // per)
        offs = np.array([(l % ring) * per for l in range(len(sizes))] + [ring * per])
        host_bytes = ring * per
    host, release, kind = pinned_host_buffer(int(host_bytes))
    if host is None:
        return {"unavailable": kind}
    try:
        tdt = torch.bfloat16 if run.w.dtype == bc.DTYPE_BF16 else torch.float32
        L = len(run.numels)
        link = link_probe(host, host_bytes)          # before the buffer is filled
        hviews = [torch.from_numpy(host[offs[l]:offs[l] + sizes[l]]).view(tdt) for l in range(L)]
        newest = bc.bc_cache_slot_ptrs(run.h, 0, L)
        for l, n in enumerate(run.numels):
            hviews[l].copy_(device_view(newest[l], n, run.w.dtype).view(tdt))
        torch.cuda.synchronize()
        # at most 16 chunks: a cache of thousands of small tensors moves in spans, not in
        # thousands of copies and calls
        cl = run.window if run.window < run.n_feat else max(chunk_layers, -(-L // 16))
        ring_mode = host_bytes < total
        ring = int(host_bytes // max(sizes)) if ring_mode else 0
        if ring_mode:
            # chunks of a divisor of the ring, at most half of it: chunk c's layers take ring
            # positions (c % regions) * cl onwards, so consecutive chunks use disjoint host
            # buffers and one chunk's copies overlap the next one's (a ring of one layer
            # leaves one chunk at a time)
            limit = min(chunk_layers, ring // 2, run.window)
            divisors = [d for d in range(1, limit + 1) if ring % d == 0]
            cl = divisors[-1] if divisors else 1
        chunks = [list(range(c, min(c + cl, L))) for c in range(0, L, cl)]
        regions = ring // cl if ring_mode else len(chunks)
        region_of = [c % regions for c in range(len(chunks))]
        pipelined = not ring_mode or ring >= 2
        s_in, s_fc, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        done_out = [None] * len(chunks)
        done_region = [None] * regions      # last read-back out of each host region
        shared_outs = run.window < run.n_feat

        slot_offs = bc.bc_cache_layout(run.h, L)

        def out_of(l, ls):
            return run.outs[l - ls[0] if shared_outs else l]

        def spans(ls, dev_addr):
            """Runs of consecutive layers of `ls` contiguous both in the host buffer and at
            the device addresses dev_addr(l): (first layer, elements)."""
            out, l0, n = [], ls[0], run.numels[ls[0]]
            for l in ls[1:]:
                if (offs[l] == offs[l - 1] + sizes[l - 1] and
                        dev_addr(l) == dev_addr(l - 1) + sizes[l - 1]):
                    n += run.numels[l]
                else:
                    out.append((l0, n))
                    l0, n = l, run.numels[l]
            out.append((l0, n))
            return out

        in_spans = [spans(ls, lambda l: slot_offs[l]) for ls in chunks]
        out_spans = [[(l0, n, out_of(l0, ls).data_ptr()) for l0, n in
                      spans(ls, lambda l, ls=ls: out_of(l, ls).data_ptr())] for ls in chunks]
        chunk_ptrs = []
        for ls in chunks:
            a = np.zeros(L, dtype=np.uint64)
            for l in ls:
                a[l] = out_of(l, ls).data_ptr()
            chunk_ptrs.append(a)

        def h2d(c, slots):
            for l0, n in in_spans[c]:
                device_view(slots[l0], n, run.w.dtype).view(tdt).copy_(
                    torch.from_numpy(host[offs[l0]:offs[l0] + n * eb]).view(tdt),
                    non_blocking=True)

        def d2h(c):
            for l0, n, ptr in out_spans[c]:
                torch.from_numpy(host[offs[l0]:offs[l0] + n * eb]).view(tdt).copy_(
                    device_view(ptr, n, run.w.dtype).view(tdt), non_blocking=True)

        def one_step_serial(i):
            # A one-layer host ring: upload, forecast and read back one chunk at a time, in
            # order on one stream, so no host buffer is read while it is being written.
            t_full, t_target = _continuation(run, i)
            slots = bc.bc_cache_next_slot_ptrs(run.h, L)
            bc.bc_cache_commit(run.h, t_full)
            with torch.cuda.stream(s_fc):
                for c, ls in enumerate(chunks):
                    h2d(c, slots)
                    bc.bc_forecast(run.h, t_target, chunk_ptrs[c], run.out_dtype,
                                   s_fc.cuda_stream)
                    d2h(c)
                ev = torch.cuda.Event()
                ev.record(s_fc)
                done_out[-1] = ev

        def one_step_ring(i):
            # Layers share host buffers: per chunk, the upload waits for the last read-back
            # out of its host region (an earlier chunk of this step or the last step), then
            # the forecast and the read-back follow on their own streams, so the next
            # chunk's upload (another region) overlaps them.
            t_full, t_target = _continuation(run, i)
            slots = bc.bc_cache_next_slot_ptrs(run.h, L)
            bc.bc_cache_commit(run.h, t_full)
            for c, ls in enumerate(chunks):
                g = region_of[c]
                with torch.cuda.stream(s_in):
                    if done_region[g] is not None:
                        s_in.wait_event(done_region[g])
                    h2d(c, slots)
                    landed = torch.cuda.Event()
                    landed.record(s_in)
                s_fc.wait_event(landed)
                if shared_outs:   # the window's output buffers are reused by every chunk
                    prev = done_out[c - 1] if c > 0 else done_out[-1]
                    if prev is not None:
                        s_fc.wait_event(prev)
                bc.bc_forecast(run.h, t_target, chunk_ptrs[c], run.out_dtype, s_fc.cuda_stream)
                ev = torch.cuda.Event()
                ev.record(s_fc)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(ev)
                    d2h(c)
                    ev2 = torch.cuda.Event()
                    ev2.record(s_out)
                    done_out[c] = ev2
                    done_region[g] = ev2

        def one_step(i):
            if ring_mode:
                return one_step_ring(i) if pipelined else one_step_serial(i)
            t_full, t_target = _continuation(run, i)
            slots = bc.bc_cache_next_slot_ptrs(run.h, L)
            landed = []
            for c, ls in enumerate(chunks):
                with torch.cuda.stream(s_in):
                    if done_out[c] is not None:
                        s_in.wait_event(done_out[c])
                    h2d(c, slots)
                    ev = torch.cuda.Event()
                    ev.record(s_in)
                    landed.append(ev)
            bc.bc_cache_commit(run.h, t_full)
            for c, ls in enumerate(chunks):
                s_fc.wait_event(landed[c])
                if shared_outs:   # the window's output buffers are reused by every chunk
                    prev = done_out[c - 1] if c > 0 else done_out[-1]
                    if prev is not None:
                        s_fc.wait_event(prev)
                bc.bc_forecast(run.h, t_target, chunk_ptrs[c], run.out_dtype, s_fc.cuda_stream)
                ev = torch.cuda.Event()
                ev.record(s_fc)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(ev)
                    d2h(c)
                    ev2 = torch.cuda.Event()
                    ev2.record(s_out)
                    done_out[c] = ev2

        one_step(0)                      # warm-up
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        t0 = time.perf_counter()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        marks = []
        a.record()
        for i in range(steps):
            one_step(i + 1)
            ev = torch.cuda.Event(enable_timing=True)      # this step's last read-back
            ev.record(s_out if pipelined else s_fc)
            marks.append(ev)
        for ev in done_out:
            if ev is not None:
                torch.cuda.current_stream().wait_event(ev)
        b.record()
        torch.cuda.synchronize()
        step_marks = [round(a.elapsed_time(m), 1) for m in marks]
        wall = time.perf_counter() - t0
        ms = max_over_ranks(a.elapsed_time(b) / steps, dist)
        alg = run.algorithmic_bytes()
        moved = total + run.n_feat * run.w.layer_numel * ob
        link_gbs = moved / (ms * 1e-3) / 1e9
        return {"value": round(job_throughput(alg, ms, world), 1), "unit": "GB/s",
                "h2d_bytes_per_step": total,
                "d2h_bytes_per_step": run.n_feat * run.w.layer_numel * ob,
                "host_link_GB/s": round(link_gbs, 1),
                "step_end_ms": step_marks,
                "link_probe": link,
                "frac_of_link_both": (round(link_gbs / link["both_GB/s"], 3)
                                      if link and link.get("both_GB/s") else None),
                "ms_per_step": round(ms, 3), "wall_s": round(wall, 3), "steps": steps,
                "chunk_layers": cl, "host_memory": kind, "host_buffer_bytes": int(host_bytes),
                "overlapped": pipelined,
                "host_ring_layers": ring or None,
                "path": "pinned host -> next cache slot (bc_cache_next_slot_ptrs + "
                        "bc_cache_commit) -> bc_forecast per chunk -> pinned host, " +
                        ("pipelined over 3 streams" if not ring_mode else
                         f"pipelined over 3 streams through a ring of {ring} layers of host "
                         "buffers (page-locked memory capped per rank)" if pipelined else
                         "one chunk at a time on one stream (host buffers shared by layers)")}
    finally:
        torch.cuda.synchronize()
        release()


CHUNK = 1 << 22   # elements per oracle call in the CPU samples


def _oracle_pool_init():
    import oracle
    oracle.build()
    oracle._load()


def _oracle_task(args):
    """One oracle call on a chunk held in shared memory (runs in a spawned worker)."""
    from multiprocessing import shared_memory
    import numpy as np
    import oracle
    shm_name, dtype, m, total, off, size, W = args
    shm = shared_memory.SharedMemory(name=shm_name)
    try:
        arr = np.ndarray((m, total), dtype=dtype, buffer=shm.buf)
        F = [arr[j, off:off + size] for j in range(m)]
        oracle.combine(F, W)
        del F, arr
    finally:
        shm.close()
    return size


class OraclePool:
    """The unmodified fp64 oracle on every host core: a spawn pool of one worker per core,
    each running oracle.combine on chunks of a sample held in shared memory.  `capacity`
    (elements per node) sizes the shared block for later samples given to load()."""

    def __init__(self, sample: list, W, workers: int | None = None,
                 capacity: int | None = None):
        import multiprocessing as mp
        from multiprocessing import shared_memory
        self.m = len(sample)
        self.dtype = sample[0].dtype
        self.capacity = max(capacity or 0, sample[0].size)
        self.shm = shared_memory.SharedMemory(
            create=True, size=max(1, self.m * self.capacity * sample[0].itemsize))
        self.W = [float(w) for w in W]
        self.workers = workers or os.cpu_count() or 1
        self.pool = mp.get_context("spawn").Pool(self.workers, initializer=_oracle_pool_init)
        self.load(sample)
        self.pool.map(_oracle_task, self.tasks[:self.workers])        # warm the workers

    def load(self, sample: list):
        """Copy a new sample (same node count and dtype, at most `capacity` elements per
        node) into the shared block."""
        import numpy as np
        assert len(sample) == self.m and sample[0].dtype == self.dtype
        total = sample[0].size
        assert total <= self.capacity
        arr = np.ndarray((self.m, self.capacity), dtype=self.dtype, buffer=self.shm.buf)
        for j in range(self.m):
            arr[j, :total] = sample[j]
        del arr
        self.total = total
        self.tasks = [(self.shm.name, self.dtype, self.m, self.capacity, off,
                       min(CHUNK, total - off), self.W)
                      for off in range(0, total, CHUNK)]

    def run(self, passes: int = 1):
        """Process the whole sample `passes` times; returns (elements, seconds)."""
        t0 = time.perf_counter()
        done = sum(sum(self.pool.map(_oracle_task, self.tasks, chunksize=1))
                   for _ in range(passes))
        return done, time.perf_counter() - t0

    def close(self):
        self.pool.close()
        self.pool.join()
        self.shm.close()
        self.shm.unlink()


def _time_oracle(chunks, W, seconds):
    """Time the oracle over host chunks (list of lists of K arrays) until `seconds` pass or
    the chunks run out; returns (elements, seconds)."""
    import oracle
    done, spent = 0, 0.0
    for F in chunks:
        t0 = time.perf_counter()
        oracle.combine(F, W)
        spent += time.perf_counter() - t0
        done += F[0].size
        if spent >= seconds:
            break
    return done, spent


def host_info():
    """The host the CPU legs ran on: architecture, CPU model (lscpu, when present) and the
    number of online cores."""
    import platform
    info = {"machine": platform.machine(), "nproc": os.cpu_count()}
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            key, _, val = line.partition(":")
            if key.strip() in ("Model name", "Vendor ID", "Socket(s)", "NUMA node(s)"):
                info[key.strip()] = val.strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return info


def cpu_baseline_from_device(run, seconds):
    """The fp64 oracle on the host over a bounded sample of the same workload: 64 chunks of
    4 Mi consecutive elements of the live history slots (copied to the host first, outside
    the timed region; layers round-robin; 1.5 GB of bf16, far beyond the host caches).  Timed
    on every host core (spawned workers running the unmodified oracle) and, for reference, on
    one core."""
    import numpy as np
    import oracle
    from paper_2608_28670_gb300.runner import device_view

    p = run.problem
    W = oracle.paper_weights(list(p.nodes), p.t)
    m = len(p.nodes)
    slots = [bc_slot_ptrs(run, j) for j in range(m)]
    n_chunks = 64
    parts = [[] for _ in range(m)]
    for c in range(n_chunks):
        l = c % run.n_feat
        n = run.numels[l]
        size = min(CHUNK, n)
        off = ((c * 2654435761) % max(1, n - size + 1)) // 8 * 8
        for j in range(m):
            v = device_view(slots[j][l], n, run.w.dtype)[off:off + size].cpu().numpy()
            parts[j].append(v.view(np.uint16) if v.dtype == np.int16 else v)
    sample = [np.concatenate(parts[j]) for j in range(m)]
    per_elem = run.algorithmic_bytes() / (run.w.layer_numel * run.n_feat)

    # one core
    one = [[sample[j][o:o + CHUNK] for j in range(m)] for o in range(0, sample[0].size, CHUNK)]
    n1, t1 = _time_oracle(one, W, seconds / 3)
    # every core
    pool = OraclePool(sample, W)
    try:
        e0, s0 = pool.run(1)
        passes = max(1, int((2 * seconds / 3) / max(s0, 1e-3)))
        e1, s1 = pool.run(passes)
        elems, secs = e0 + e1, s0 + s1
        cores = pool.workers
    finally:
        pool.close()
    step_elems = run.w.layer_numel * run.n_feat
    return {"value": round(elems * per_elem / secs / 1e9, 4), "unit": "GB/s", "cores": cores,
            "kind": "oracle", "elems_per_s": round(elems / secs, 1),
            "sample": f"{sample[0].size} elements ({n_chunks} chunks of "
                      f"{max(x.size for x in parts[0])} consecutive elements, "
                      f"layers round-robin) of the K={m} history slots, processed {1 + passes} "
                      f"times by {cores} spawned workers running the fp64 oracle, {secs:.1f} s",
            "whole_step_s": round(step_elems / (elems / secs), 1),
            "whole_step_s_is": f"extrapolated: the step's {step_elems} elements at the "
                               f"sample's rate",
            "host": host_info(),
            "single_core": {"value": round(n1 * per_elem / t1 / 1e9, 4), "cores": 1,
                            "elems_per_s": round(n1 / t1, 1), "seconds": round(t1, 1),
                            "whole_step_s": round(step_elems / (n1 / t1), 1)}}


GROUP_ELEMS = 1 << 27   # elements per node copied to the host at a time (full baselines)


def _host_slot(ptr, n, dtype):
    """Host copy of n stored elements at a device address (bf16 as uint16 words)."""
    import numpy as np
    from paper_2608_28670_gb300.runner import device_view
    v = device_view(ptr, n, dtype).cpu().numpy()
    return v.view(np.uint16) if v.dtype == np.int16 else v


def cpu_baseline_full(run, min_seconds=0.5):
    """The unmodified fp64 oracle over every element of the workload: each layer's forecast
    from its live history slots (and on the sampler layer the Euler update), on one core and
    on every core (spawned workers).  Layers are copied to the host in groups of about
    GROUP_ELEMS elements per node outside the timed regions; only oracle calls are timed.  A
    workload that takes less than `min_seconds` on one core is processed repeatedly."""
    import numpy as np
    import oracle
    p = run.problem
    W = oracle.paper_weights(list(p.nodes), p.t)
    m = len(p.nodes)
    slots = [bc_slot_ptrs(run, j) for j in range(m)]
    groups, cur, n_cur = [], [], 0
    for l in range(run.n_feat):
        n = run.numels[l]
        if cur and n_cur + n > GROUP_ELEMS:
            groups.append(cur)
            cur, n_cur = [], 0
        cur.append(l)
        n_cur += n
    if cur:
        groups.append(cur)
    cap = max(sum(run.numels[l] for l in g) for g in groups)
    one_s = all_s = 0.0
    elems = 0
    pool = None
    passes = 1
    try:
        for gi, g in enumerate(groups):
            F = [np.concatenate([_host_slot(slots[j][l], run.numels[l], run.w.dtype)
                                 for l in g]) for j in range(m)]
            chunks = [[f[o:o + CHUNK] for f in F] for o in range(0, F[0].size, CHUNK)]
            if gi == 0:
                t0 = time.perf_counter()
                for c in chunks:
                    oracle.combine(c, W)
                first = time.perf_counter() - t0
                if len(groups) == 1 and first < min_seconds:
                    passes = max(1, int(min_seconds / max(first, 1e-6)))
            t0 = time.perf_counter()
            for _ in range(passes):
                for c in chunks:
                    oracle.combine(c, W)
            one_s += time.perf_counter() - t0
            if pool is None:
                pool = OraclePool(F, W, capacity=cap)
            else:
                pool.load(F)
            _, secs = pool.run(passes)
            all_s += secs
            elems += F[0].size
            del F, chunks
        if run.euler:
            l = len(run.numels) - 1
            V = [_host_slot(slots[j][l], run.numels[l], run.w.dtype) for j in range(m)]
            x = run.x.cpu().numpy()
            t0 = time.perf_counter()
            for _ in range(passes):
                oracle.euler(V, W, x, p.dt)
            te = time.perf_counter() - t0
            one_s += te
            all_s += te
            elems += V[0].size
        cores = pool.workers
    finally:
        if pool is not None:
            pool.close()
    alg = run.algorithmic_bytes() * passes
    return {"value": round(alg / all_s / 1e9, 4), "unit": "GB/s", "cores": cores,
            "kind": "oracle", "elems_per_s": round(elems * passes / all_s, 1),
            "seconds": round(all_s, 3),
            "sample": f"the whole workload: {elems} elements ({run.n_feat} layers"
                      f"{' + the Euler layer' if run.euler else ''}, K={m}), "
                      f"{passes} pass(es), fp64 oracle on {cores} spawned workers"
                      f"{'; the Euler layer on one core' if run.euler else ''}",
            "single_core": {"value": round(alg / one_s / 1e9, 4), "cores": 1,
                            "elems_per_s": round(elems * passes / one_s, 1),
                            "seconds": round(one_s, 3)}}


def bc_slot_ptrs(run, j):
    from paper_2608_28670_gb300 import barycache as bc
    return bc.bc_cache_slot_ptrs(run.h, j, len(run.numels))


def run_reference(args):
    """The oracle as the reference arm: fp64, single-threaded, on the host cores, on a
    bounded host-generated sample of the same workload per step."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    import oracle
    from paper_2608_28670_gb300 import synth
    from paper_2608_28670_gb300.configs import WORKLOADS
    oracle.build()
    w = WORKLOADS[args.workload]
    K = args.K or w.K
    p = w.representative(K)
    n = 1 << 25                       # 32 Mi elements per node: inputs beyond the host L3
    nodes_oldest_first = list(reversed(p.nodes))
    feats = synth.host_trajectories([(n,)], [w.tau(t) for t in nodes_oldest_first],
                                    dtype="bf16" if w.elem_bytes == 2 else "f32",
                                    degree=w.degree, noise_std=w.noise_std, seed=2026)
    F = [f[0] for f in reversed(feats)]        # newest first
    W = oracle.paper_weights(list(p.nodes), p.t)
    per_elem = (K * w.elem_bytes + w.elem_bytes)
    pool = OraclePool(F, W)
    try:
        for _ in range(args.warmup):
            pool.run(1)
        times = []
        for _ in range(args.steps):
            _, secs = pool.run(1)
            times.append(secs)
        cores = pool.workers
    finally:
        pool.close()
    ms = 1e3 * sum(times) / len(times)
    value = n * per_elem / (ms * 1e-3) / 1e9
    sample = (f"{n} elements per step of one [{n}] slice at K={K} (host-generated with the "
              f"workload's recipe), fp64 oracle on {cores} spawned workers")
    out = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": w.name, "K": K, "nodes": list(p.nodes), "target": p.t,
                      "sample_elements_per_step": n},
           "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": cores,
                            "kind": "oracle", "sample": sample, "host": host_info()},
           "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()

#!/usr/bin/env python3
"""Benchmark of the GB300 hot path (isam C ABI) -- one JSON line on rank 0.

Timed workload (one "step"): the tall-skinny GEMM sweep of the paper's
DeepBench-sized GEMM benchmark (Section 5.1.1): (M, K) in {(1760,1760),
(2560,2560), (4096,4096), (7680,2560)} x N in {16, 32, 64, 128} x {NN, TN},
bf16 operands U[-1,1], fp32 accumulate and output, beta = 0.  32 GEMMs per
step, each on its own operands (0.78 GB per step, larger than L2, so no
GEMM finds its operands in L2 from the step before).  A step is one
isam_gemm_grouped call over the 32 problems (one persistent launch).

value  = GEMM TFLOP/s over the sweep (all ranks' flops / max rank time).
e2e    = the same through host buffers (two device operand sets, so one step's
         input copies overlap the previous step's GEMM): pinned host -> device copies of every
         operand, the grouped call, device -> host copies of every result.
roofline: the sweep's kernel (gemm_group_kernel) is HBM-bound: algorithmic
         bytes (2MK + 2KN + 4MN per GEMM, summed) / per-launch CUDA-event time,
         against the measured copy bandwidth.
per_call_sweep: the same 32 GEMMs as 32 isam_gemm calls (one launch each).
hot_path: the other rows measured in the same run (not part of value): the
         8192^3 GEMM with beta = 1 (TFLOP/s vs dense bf16), the GRU forward
         (hidden 1024, batch 32, 128 steps: timesteps/s), the fused separable
         depthwise layer (32x56x56, 128 -> 256: GB/s vs HBM).
cpu_baseline: the fp64 oracle on the host cores, on a row sample of the sweep.

--impl reference times the oracle itself (the paper publishes no code to run
instead) on the same workload's row sample, K steps after W warm-up steps.
Multi-GPU (torchrun): every rank runs the whole sweep on its own GPU with no
collective on the data path (weak scaling); timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

SWEEP_MK = [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)]
SWEEP_N = [16, 32, 64, 128]
METRIC = "GEMM TFLOP/s (tall-skinny sweep) and GRU timesteps/s on 1 GB300; % of roofline"
WORKLOAD = ("tall-skinny GEMM sweep: (M,K) in {(1760,1760),(2560,2560),(4096,4096),(7680,2560)} "
            "x N in {16,32,64,128} x {NN,TN}; bf16 U[-1,1]; fp32 accumulate/output; beta=0")
# dram__bytes_read.sum + dram__bytes_write.sum of one gemm_group_kernel launch
# over the sweep (749995520 + 24220928 bytes), from an ncu capture of the kernel
# with 256-row tiles for the heavy problems, per-tile register copies of the
# problem fields and C stored straight from TMEM; None whenever the kernel
# changes until the counters are taken again.
TRAFFIC_PER_STEP = 774216448
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# --------------------------------------------------------------------------- host logic
def sweep_config(world: int) -> dict:
    """The workload description both arms print (identical keys and values)."""
    bytes_step = sum(gemm_bytes(M, N, K) for (M, N, K, _t) in sweep_problems())
    return {"workload": WORKLOAD, "gemms_per_step": 32,
            "l2": "inputs larger than L2: each GEMM has its own operands, "
                  f"{bytes_step / 1e9:.2f} GB per step",
            "parallelism": f"replica x{world}"}


def sweep_problems():
    """(M, N, K, transA) of the 32 GEMMs of one step, in launch order."""
    return [(M, N, K, tA) for tA in (0, 1) for (M, K) in SWEEP_MK for N in SWEEP_N]


def gemm_flops(M, N, K):
    return 2.0 * M * N * K


def gemm_bytes(M, N, K, beta=False):
    return 2.0 * M * K + 2.0 * K * N + 4.0 * M * N * (2 if beta else 1)


def whole_job_tflops(flops_per_step: float, steps: int, world: int, max_rank_ms: float) -> float:
    """All ranks' flops over the slowest rank's time (every rank runs the full
    step: weak scaling)."""
    return flops_per_step * steps * world / (max_rank_ms / 1e3) / 1e12


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def reduce_max(x: float, backend_device=None) -> float:
    """Max of a float over all ranks (identity without torch.distributed)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=backend_device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def row_sample(M: int, stride: int):
    import numpy as np
    return np.arange(0, M, stride, dtype=np.int32)


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampled every 5 ms in the background."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.rows = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "5"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return self
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), [c.strip() for c in line.split(",")]))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            if self.thread:
                self.thread.join(timeout=2)

    def summary(self, t0: float, t1: float):
        inside = [r for (t, r) in self.rows if t0 <= t <= t1]
        window = "timed"
        if not inside and self.rows:
            mid = 0.5 * (t0 + t1)
            inside = [min(self.rows, key=lambda tr: abs(tr[0] - mid))[1]]
            window = "nearest"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(r[1]) for r in inside if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in inside if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i in range(4)
                          if len(r) > 5 + i and r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(inside), "window": window}


# --------------------------------------------------------------------------- GPU arm
def make_sweep(dev):
    import torch
    from paper_1810_09958_gb300 import synth
    probs = []
    for (M, N, K, tA) in sweep_problems():
        seed = synth.stream_seed(synth.BASE_SEED, 1, M, K, N, tA)
        A = synth.bf16_uniform_torch(synth.stream_seed(seed, 1), M * K, dev)
        B = synth.bf16_uniform_torch(synth.stream_seed(seed, 2), K * N, dev)
        C = torch.empty(M * N, dtype=torch.float32, device=dev)
        probs.append({"M": M, "N": N, "K": K, "tA": tA, "A": A, "B": B, "C": C,
                      "flops": gemm_flops(M, N, K), "bytes": gemm_bytes(M, N, K)})
    return probs


def run_sweep(isam, probs):
    for p in probs:
        isam.gemm(p["M"], p["N"], p["K"], p["tA"], 0, 1.0, p["A"], p["B"], 0.0, p["C"])


def time_sweep(isam, probs, steps, warmup):
    """K steps of the sweep, each one replay of a CUDA graph holding the 32
    GEMM launches (so host launch cost does not leak into microsecond kernels);
    CUDA events on the replay stream bracket the timed region."""
    import torch
    for _ in range(warmup):
        run_sweep(isam, probs)
    isam.sync()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        run_sweep(isam, probs)
    for _ in range(warmup):
        graph.replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    t0 = time.time()
    start.record(stream)
    for _ in range(steps):
        graph.replay()
    end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    barrier()
    isam.sync()
    del graph
    return start.elapsed_time(end), (t0, t1)


def time_grouped(isam, probs, steps, warmup):
    """K steps of the sweep as ONE isam_gemm_grouped launch per step (the 32
    problems share one persistent grid), replayed as a CUDA graph."""
    import torch
    call = isam.GroupedGemm([(p["M"], p["N"], p["K"], p["tA"], 0, 1.0, p["A"], p["B"], 0.0, p["C"])
                             for p in probs])
    for _ in range(warmup):
        call()
    isam.sync()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        call()
    for _ in range(warmup):
        graph.replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    t0 = time.time()
    start.record(stream)
    for _ in range(steps):
        graph.replay()
    end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    barrier()
    isam.sync()
    del graph
    return start.elapsed_time(end), (t0, t1)


def time_e2e(isam, probs, steps, warmup):
    """The sweep through host buffers: per step, the pinned host -> device copy
    of every operand, one isam_gemm_grouped launch, the device -> host copy of
    every result.  Each step's operands sit back to back in one pinned host
    buffer and one device buffer (likewise the results), so a step moves them
    in one copy each way.  Steps alternate between two device operand sets so
    that the input copy of step k + 1 (copy stream) overlaps the GEMM and the
    result copy of step k; events order each set's copies, GEMM and read-back,
    and every step still moves its own inputs in and its result out."""
    import torch

    def layout(sizes):
        offs, at = [], 0
        for n in sizes:
            offs.append(at)
            at += (n + 255) // 256 * 256
        return offs, at

    in_sizes = []
    for p in probs:
        in_sizes += [p["A"].numel() * 2, p["B"].numel() * 2]
    in_offs, in_total = layout(in_sizes)
    out_offs, out_total = layout([p["M"] * p["N"] * 4 for p in probs])
    host_in = torch.empty(in_total, dtype=torch.uint8).pin_memory()
    host_out = torch.empty(out_total, dtype=torch.uint8).pin_memory()
    for j, p in enumerate(probs):
        for t, name in ((2 * j, "A"), (2 * j + 1, "B")):
            host_in[in_offs[t]:in_offs[t] + in_sizes[t]].copy_(p[name].cpu().view(torch.uint8))
    h2d, d2h = in_total, out_total  # the bytes each step's two copies move
    dev_in = [torch.empty(in_total, dtype=torch.uint8, device=probs[0]["A"].device) for _ in range(2)]
    dev_out = [torch.empty(out_total, dtype=torch.uint8, device=probs[0]["A"].device) for _ in range(2)]

    def views(buf_in, buf_out):
        out = []
        for j, p in enumerate(probs):
            a0, b0 = in_offs[2 * j], in_offs[2 * j + 1]
            out.append({"A": buf_in[a0:a0 + in_sizes[2 * j]].view(torch.bfloat16),
                        "B": buf_in[b0:b0 + in_sizes[2 * j + 1]].view(torch.bfloat16),
                        "C": buf_out[out_offs[j]:out_offs[j] + p["M"] * p["N"] * 4].view(torch.float32)})
        return out
    sets = [views(dev_in[i], dev_out[i]) for i in range(2)]
    calls = [isam.GroupedGemm([(p["M"], p["N"], p["K"], p["tA"], 0, 1.0, d["A"], d["B"], 0.0, d["C"])
                               for p, d in zip(probs, ds)]) for ds in sets]
    s_in, s_run, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = {k: [torch.cuda.Event(), torch.cuda.Event()] for k in ("in", "run", "out")}
    first = [True, True]

    def one(k):
        i = k & 1
        with torch.cuda.stream(s_in):
            if not first[i]:
                s_in.wait_event(ev["run"][i])  # set i's operands are no longer read
            dev_in[i].copy_(host_in, non_blocking=True)
            ev["in"][i].record(s_in)
        with torch.cuda.stream(s_run):
            s_run.wait_event(ev["in"][i])
            if not first[i]:
                s_run.wait_event(ev["out"][i])  # set i's results have been read back
            calls[i]()
            ev["run"][i].record(s_run)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["run"][i])
            host_out.copy_(dev_out[i], non_blocking=True)
            ev["out"][i].record(s_out)
        first[i] = False

    def join(stream):
        for s in (s_in, s_run, s_out):
            e = torch.cuda.Event()
            e.record(s)
            stream.wait_event(e)

    main = torch.cuda.current_stream()
    for k in range(warmup):
        one(k)
    torch.cuda.synchronize()
    barrier()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(main)
    for s in (s_in, s_run, s_out):
        s.wait_stream(main)
    for k in range(steps):
        one(warmup + k)
    join(main)
    end.record(main)
    torch.cuda.synchronize()
    isam.sync()
    return start.elapsed_time(end), h2d, d2h


def time_call(fn, reps, warmup, flush=None):
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        if flush is not None:
            flush.zero_()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        fn()
        b.record()
        b.synchronize()
        ts.append(a.elapsed_time(b))
    return statistics.median(ts)


def per_shape_table(isam, dev, peaks, fp8=False):
    """Each sweep shape through the per-call API (isam_gemm, or isam_gemm_fp8
    on E4M3 operands for the 16 K-major shapes): a CUDA graph of back-to-back
    calls, each on its own operand set, with enough sets that a replay moves
    at least 256 MB (twice L2), so every call reads its operands from HBM.
    Returns one row per shape: kernel time per call (CUDA events over the
    replays / calls), GB/s and the fraction of the measured HBM peak."""
    import torch
    from paper_1810_09958_gb300 import synth
    rows = []
    shapes = ([(M, N, K, 0) for (M, K) in SWEEP_MK for N in SWEEP_N] if fp8 else sweep_problems())
    for (M, N, K, tA) in shapes:
        by = (M * K + N * K + 4 * M * N) if fp8 else gemm_bytes(M, N, K)
        sets = max(2, min(64, int(256e6 // by) + 1))
        ops = []
        for i in range(sets):
            seed = synth.stream_seed(synth.BASE_SEED, 9, M, K, N, tA, i)
            if fp8:
                A = synth.e4m3_uniform_torch(synth.stream_seed(seed, 1), M * K, dev)
                B = synth.e4m3_uniform_torch(synth.stream_seed(seed, 2), N * K, dev)
            else:
                A = synth.bf16_uniform_torch(synth.stream_seed(seed, 1), M * K, dev)
                B = synth.bf16_uniform_torch(synth.stream_seed(seed, 2), K * N, dev)
            ops.append((A, B, torch.empty(M * N, dtype=torch.float32, device=dev)))
        if fp8:
            run = lambda: [isam.gemm_fp8(M, N, K, 1.0, A, B, 0.0, C) for (A, B, C) in ops]
        else:
            run = lambda: [isam.gemm(M, N, K, tA, 0, 1.0, A, B, 0.0, C) for (A, B, C) in ops]
        for _ in range(2):
            run()
        isam.sync()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            run()
        ms = time_call(g.replay, reps=10, warmup=3) / sets
        del g, ops
        gbs = by / ms / 1e6
        plan = isam.gemm_plan(M, N, K, tA, 0, 0.0) if not fp8 else None
        row = {"M": M, "N": N, "K": K, "layout": "TN" if tA else "NN", "us": round(ms * 1e3, 3),
               "gbs": round(gbs, 1), "frac_hbm": round(gbs / peaks["hbm_gbs"], 4),
               "roofline_us": round(by / peaks["hbm_gbs"] / 1e3, 3)}
        if plan:
            row["plan"] = {k: plan[k] for k in ("BN", "split", "grid", "stages")}
        rows.append(row)
    torch.cuda.empty_cache()
    return rows


def hot_path_rows(isam, dev, peaks):
    """The remaining rows of the hot path, each timed on its benchmark shape."""
    import torch
    from paper_1810_09958_gb300 import synth
    out = {}
    windows = {}

    def timed(name, fn, **kw):
        # time_call, with the wall-clock window of its timed calls kept for
        # the row's clock summary
        t0 = time.time()
        ms = time_call(fn, **kw)
        windows[name] = (t0, time.time())
        return ms
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)  # 256 MB > L2
    # 8192^3, beta = 1, N(0,1)*0.02 operands, C U[-1,1].
    n = 8192
    A = synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 2, 1), n * n, dev, 0.0, 0.02)
    B = synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 2, 2), n * n, dev, 0.0, 0.02)
    C = synth.f32_uniform_torch(synth.stream_seed(synth.BASE_SEED, 2, 3), n * n, dev)
    ms = timed("gemm_8192_beta1", lambda: isam.gemm(n, n, n, 0, 0, 1.0, A, B, 1.0, C), reps=10, warmup=3)
    tf = gemm_flops(n, n, n) / ms / 1e9
    out["gemm_8192_beta1"] = {"ms": round(ms, 4), "tflops": round(tf, 1),
                              "frac_bf16_burst": round(tf / peaks["bf16_tflops"], 4),
                              "frac_bf16_sustained": round(tf / peaks["bf16_tflops_sustained"], 4),
                              "plan": isam.gemm_plan(n, n, n, 0, 0, 1.0)}
    del A, B, C
    # The skinny sweep's 16 (M, K) x N shapes on E4M3 operands (K-major A and
    # B), one isam_gemm_fp8 launch each, replayed as a CUDA graph.
    f8 = []
    for (M, K) in SWEEP_MK:
        for N_ in SWEEP_N:
            seed = synth.stream_seed(synth.BASE_SEED, 7, M, K, N_)
            f8.append((M, N_, K, synth.e4m3_uniform_torch(synth.stream_seed(seed, 1), M * K, dev),
                       synth.e4m3_uniform_torch(synth.stream_seed(seed, 2), N_ * K, dev),
                       torch.empty(M * N_, dtype=torch.float32, device=dev)))
    run_f8 = lambda: [isam.gemm_fp8(M, N_, K, 1.0, A_, B_, 0.0, C_) for (M, N_, K, A_, B_, C_) in f8]
    for _ in range(3):
        run_f8()
    isam.sync()
    g8 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g8):
        run_f8()
    ms = timed("gemm_fp8_sweep_16", g8.replay, reps=50, warmup=3) / 1.0
    fl = sum(gemm_flops(M, N_, K) for (M, N_, K, *_r) in f8)
    by = sum(M * K + N_ * K + 4 * M * N_ for (M, N_, K, *_r) in f8)
    out["gemm_fp8_sweep_16"] = {"ms": round(ms, 4), "tflops": round(fl / ms / 1e9, 1),
                                "gbs": round(by / ms / 1e6, 1), "frac_hbm": round(by / ms / 1e6 / peaks["hbm_gbs"], 4),
                                "what": "16 skinny shapes, E4M3 A (M x K) and B (N x K), fp32 C; "
                                        "one isam_gemm_fp8 launch each (graph replay)"}
    # The same 16 problems as one isam_gemm_grouped_fp8 launch.
    gcall = isam.GroupedGemmFp8([(M, N_, K, 1.0, A_, B_, 0.0, C_) for (M, N_, K, A_, B_, C_) in f8])
    for _ in range(3):
        gcall()
    isam.sync()
    gg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gg):
        gcall()
    ms = timed("gemm_fp8_grouped_16", gg.replay, reps=50, warmup=3)
    out["gemm_fp8_grouped_16"] = {"ms": round(ms, 4), "tflops": round(fl / ms / 1e9, 1),
                                  "gbs": round(by / ms / 1e6, 1),
                                  "frac_hbm": round(by / ms / 1e6 / peaks["hbm_gbs"], 4),
                                  "what": "the same 16 E4M3 problems in one isam_gemm_grouped_fp8 launch"}
    # The same 16 shapes as block-scaled (MX) E4M3: one E8M0 scale per 32 K
    # elements of every row of A and B, one isam_gemm_grouped_mxfp8 launch.
    mx = []
    for (M, N_, K, A_, B_, C_) in f8:
        seed = synth.stream_seed(synth.BASE_SEED, 8, M, K, N_)
        SA = torch.randint(120, 135, (isam.mx_scale_bytes(M, K),), dtype=torch.uint8, device=dev,
                           generator=torch.Generator(device=dev).manual_seed(seed & 0x7FFFFFFF))
        SB = torch.randint(120, 135, (isam.mx_scale_bytes(N_, K),), dtype=torch.uint8, device=dev,
                           generator=torch.Generator(device=dev).manual_seed((seed >> 1) & 0x7FFFFFFF))
        mx.append((M, N_, K, 1.0, A_, SA, B_, SB, 0.0, C_))
    mcall = isam.GroupedGemmMxfp8(mx)
    for _ in range(3):
        mcall()
    isam.sync()
    gm = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gm):
        mcall()
    ms = timed("gemm_mx_grouped_16", gm.replay, reps=50, warmup=3)
    bym = sum(M * K + N_ * K + isam.mx_scale_bytes(M + N_, K) + 4 * M * N_ for (M, N_, K, *_r) in mx)
    out["gemm_mx_grouped_16"] = {"ms": round(ms, 4), "tflops": round(fl / ms / 1e9, 1),
                                 "gbs": round(bym / ms / 1e6, 1),
                                 "frac_hbm": round(bym / ms / 1e6 / peaks["hbm_gbs"], 4),
                                 "what": "the 16 problems as block-scaled E4M3 (E8M0 scale per 32 K elements "
                                         "of each row of A and B) in one isam_gemm_grouped_mxfp8 launch"}
    del f8, g8, gg, gcall, mx, gm, mcall
    # GRU: hidden = input = 1024, batch 32, T = 128.
    T, batch, H = 128, 32, 1024
    s = 1.0 / 32.0
    x = synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 3, 1), T * batch * H, dev)
    W = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 3, 2), 3 * H * H, dev, -s, s)
    U = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 3, 3), 3 * H * H, dev, -s, s)
    b = synth.f32_uniform_torch(synth.stream_seed(synth.BASE_SEED, 3, 4), 6 * H, dev, -0.1, 0.1)
    h0 = torch.zeros(batch * H, dtype=torch.float32, device=dev)
    hout = torch.empty(T * batch * H, dtype=torch.float32, device=dev)
    ms = timed("gru_h1024_b32_t128", lambda: isam.gru_forward(T, batch, H, x, W, U, b, h0, hout), reps=10, warmup=3,
                   flush=flush)
    gflop = 2.0 * T * batch * 3 * H * (H + H) / 1e9
    tf = gflop / ms
    out["gru_h1024_b32_t128"] = {"ms": round(ms, 4), "timesteps_per_s": round(T / (ms / 1e3), 1),
                                 "us_per_step": round(ms * 1e3 / T, 3), "tflops": round(tf, 2),
                                 "frac_bf16_burst": round(tf / peaks["bf16_tflops"], 4)}
    # The same GRU with the reset gate applied before the candidate's product
    # (two exchange rounds per step).
    ms = timed("gru_reset_before_h1024_b32_t128", lambda: isam.gru_forward(T, batch, H, x, W, U, b, h0, hout, reset_before=True),
                   reps=10, warmup=3, flush=flush)
    tf = gflop / ms
    out["gru_reset_before_h1024_b32_t128"] = {
        "ms": round(ms, 4), "timesteps_per_s": round(T / (ms / 1e3), 1),
        "us_per_step": round(ms * 1e3 / T, 3), "tflops": round(tf, 2),
        "frac_bf16_burst": round(tf / peaks["bf16_tflops"], 4)}
    del x, W, U, b, h0, hout
    # Two stacked layers (one persistent kernel advancing both, the upper
    # layer's projection computed from the lower layer's tiles), against the
    # same stack as one call per layer.
    L = 2
    x = synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 5, 1), T * batch * H, dev)
    W = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 5, 2), L * 3 * H * H, dev, -s, s)
    U = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 5, 3), L * 3 * H * H, dev, -s, s)
    b = synth.f32_uniform_torch(synth.stream_seed(synth.BASE_SEED, 5, 4), L * 6 * H, dev, -0.1, 0.1)
    hout = torch.empty(L * T * batch * H, dtype=torch.float32, device=dev)
    ms = timed("gru_stack2_h1024_b32_t128", lambda: isam.gru_forward_stack(L, T, batch, H, x, W, U, b, None, hout), reps=10,
                   warmup=3, flush=flush)
    seq = T * batch * H
    x1 = torch.empty(seq, dtype=torch.bfloat16, device=dev)

    def per_layer():
        isam.gru_forward(T, batch, H, x, W[:3 * H * H], U[:3 * H * H], b[:6 * H], None, hout[:seq])
        x1.copy_(hout[:seq])
        isam.gru_forward(T, batch, H, x1, W[3 * H * H:], U[3 * H * H:], b[6 * H:], None, hout[seq:])
    ms_pl = timed("gru_stack2_per_layer", per_layer, reps=10, warmup=3, flush=flush)
    out["gru_stack2_h1024_b32_t128"] = {
        "ms": round(ms, 4), "layer_timesteps_per_s": round(L * T / (ms / 1e3), 1),
        "us_per_layer_step": round(ms * 1e3 / (L * T), 3),
        "per_layer_calls_ms": round(ms_pl, 4),
        "what": "2 layers in one isam_gru_forward_stack call (both layers in one kernel); "
                "per_layer_calls_ms: two isam_gru_forward calls with a bf16 cast (torch) between"}
    del x, W, U, b, hout, x1
    # Separable depthwise layer.
    N, Hh, Ww, Cin, Cout = 32, 56, 56, 128, 256
    xd = synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 4, 1), N * Hh * Ww * Cin, dev)
    dw = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 4, 2), 9 * Cin, dev, -1 / 3, 1 / 3)
    pw = synth.bf16_uniform_torch(synth.stream_seed(synth.BASE_SEED, 4, 3), Cin * Cout, dev,
                                  -Cin ** -0.5, Cin ** -0.5)
    od = torch.empty(N * Hh * Ww * Cout, dtype=torch.float32, device=dev)
    ms = timed("dwsep_32x56x56_128_256", lambda: isam.dwsep_conv(N, Hh, Ww, Cin, Cout, xd, dw, pw, od), reps=20, warmup=3,
                   flush=flush)
    byts = N * Hh * Ww * (Cin * 2 + Cout * 4) + 9 * Cin * 2 + Cin * Cout * 2
    gbs = byts / ms / 1e6
    # The same layer sustained: a CUDA graph of calls on 8 operand sets in
    # turn (1 GB per replay, so every call reads its input from HBM, and each
    # call's output is written back while later calls run), per call.
    sets = 8
    xs = [synth.bf16_normal_torch(synth.stream_seed(synth.BASE_SEED, 4, 10 + i), N * Hh * Ww * Cin, dev)
          for i in range(sets)]
    ods = [torch.empty(N * Hh * Ww * Cout, dtype=torch.float32, device=dev) for _ in range(sets)]
    run_sets = lambda: [isam.dwsep_conv(N, Hh, Ww, Cin, Cout, xs[i], dw, pw, ods[i]) for i in range(sets)]
    run_sets()
    isam.sync()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        run_sets()
    ms_rot = timed("dwsep_32x56x56_128_256_rotating", graph.replay, reps=10, warmup=3) / sets
    del graph
    out["dwsep_32x56x56_128_256"] = {"ms": round(ms, 4), "gbs": round(gbs, 1),
                                     "frac_hbm": round(gbs / peaks["hbm_gbs"], 4),
                                     "tflops": round(2.0 * N * Hh * Ww * Cin * (9 + Cout) / ms / 1e9, 2),
                                     "ms_rotating": round(ms_rot, 4),
                                     "frac_hbm_rotating": round(byts / ms_rot / 1e6 / peaks["hbm_gbs"], 4),
                                     "what": "ms: one call after an L2 flush (a 256 MB write); ms_rotating: per call "
                                             "of a graph of 8 calls on 8 operand sets (1 GB per replay)"}
    # The same layer unfused: the depthwise factor to memory (bf16), then the
    # pointwise factor through isam_gemm (M = N*H*W, N = Cout, K = Cin).
    M = N * Hh * Ww
    yb = torch.empty(M * Cin, dtype=torch.bfloat16, device=dev)
    ms_dw = timed("dwsep_unfused_depthwise", lambda: isam.depthwise_conv3x3(N, Hh, Ww, Cin, xd, dw, yb), reps=20,
                  warmup=3, flush=flush)
    ms_pw = timed("dwsep_unfused_pointwise", lambda: isam.gemm(M, Cout, Cin, 0, 0, 1.0, yb, pw, 0.0, od), reps=20,
                  warmup=3, flush=flush)

    def unfused():
        isam.depthwise_conv3x3(N, Hh, Ww, Cin, xd, dw, yb)
        isam.gemm(M, Cout, Cin, 0, 0, 1.0, yb, pw, 0.0, od)
    ms_u = timed("dwsep_unfused_32x56x56_128_256", unfused, reps=20, warmup=3, flush=flush)
    bytes_u = byts + 2 * M * Cin * 2  # the intermediate written and read back

    def unfused_sets():
        for i in range(sets):
            isam.depthwise_conv3x3(N, Hh, Ww, Cin, xs[i], dw, yb)
            isam.gemm(M, Cout, Cin, 0, 0, 1.0, yb, pw, 0.0, ods[i])
    unfused_sets()
    isam.sync()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        unfused_sets()
    ms_urot = timed("dwsep_unfused_32x56x56_128_256_rotating", graph.replay, reps=10, warmup=3) / sets
    del graph, xs, ods
    out["dwsep_unfused_32x56x56_128_256"] = {
        "ms": round(ms_u, 4), "depthwise_ms": round(ms_dw, 4), "pointwise_ms": round(ms_pw, 4),
        "gbs": round(bytes_u / ms_u / 1e6, 1), "frac_hbm": round(bytes_u / ms_u / 1e6 / peaks["hbm_gbs"], 4),
        "layer_gbs": round(byts / ms_u / 1e6, 1), "ms_rotating": round(ms_urot, 4),
        "what": "isam_depthwise_conv3x3 (bf16 intermediate in HBM) then isam_gemm; gbs counts the intermediate's "
                "round trip, layer_gbs the fused layer's algorithmic bytes"}
    isam.sync()
    return out, windows


# --------------------------------------------------------------------------- CPU (oracle) arm
def sample_operands(stride):
    """Every stride-th row i of op(A) of each sweep GEMM, with its full B, drawn
    from the same streams as the GPU arm's operands (the generator is
    counter-based, so only the sampled entries are drawn).  Row r of the
    returned A_sub is row rows[r] of op(A); the oracle then computes exactly
    rows[r] of C as a (len(rows) x N x K) problem."""
    import numpy as np
    from paper_1810_09958_gb300 import synth
    ops = []
    for (M, N, K, tA) in sweep_problems():
        seed = synth.stream_seed(synth.BASE_SEED, 1, M, K, N, tA)
        rows = row_sample(M, stride).astype(np.uint64)
        ks = np.arange(K, dtype=np.uint64)
        idx = (ks[None, :] * np.uint64(M) + rows[:, None]) if tA else (rows[:, None] * np.uint64(K) + ks[None, :])
        A_sub = synth.to_bf16_bits(synth.uniform_at(synth.stream_seed(seed, 1), idx))
        B = synth.bf16_uniform(synth.stream_seed(seed, 2), (K, N))
        ops.append((rows.size, N, K, A_sub, B))
    return ops


def oracle_sample_run(ops):
    """The oracle on a row sample of every sweep GEMM; returns (seconds, flops)."""
    import oracle
    t0 = time.perf_counter()
    flops = 0.0
    for (R, N, K, A_sub, B) in ops:
        oracle.gemm(R, N, K, 0, 0, 1.0, A_sub, B)
        flops += 2.0 * R * N * K
    return time.perf_counter() - t0, flops


def full_pass_seconds():
    """Oracle time of one full pass over the sweep, extrapolated from a
    stride-64 row sample."""
    probe = 64
    t, _ = oracle_sample_run(sample_operands(probe))
    return t * probe


def stride_for(target_s, t_full):
    return max(1, int(round(t_full / max(target_s, 1e-3))))


def cpu_baseline(target_s=12.0):
    """The oracle as it stands on this host's cores: a row sample of the sweep
    (all rows when a full pass is short), repeated to about target_s."""
    import oracle
    t_full = full_pass_seconds()
    stride = stride_for(target_s, t_full)
    ops = sample_operands(stride)
    reps = max(1, int(round(target_s / max(t_full / stride, 1e-3)))) if stride == 1 else 1
    t, flops = 0.0, 0.0
    for _ in range(reps):
        dt, df = oracle_sample_run(ops)
        t += dt
        flops += df
    rows = "all rows" if stride == 1 else f"every {stride}th row"
    return {"value": flops / t / 1e12, "unit": "TFLOP/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"fp64 oracle, {rows} of each of the 32 sweep GEMMs, {reps} pass(es): "
                      f"{flops / 1e9:.2f} GFLOP in {t:.1f} s"}


def reference_arm(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    # Each step a row sample sized so that all W + K steps take about two minutes.
    t_full = full_pass_seconds()
    per_step = min(4.0, 120.0 / max(1, args.steps + args.warmup))
    stride = stride_for(per_step, t_full)
    ops = sample_operands(stride)
    warm = sample_operands(stride * 8)
    for _ in range(args.warmup):
        oracle_sample_run(warm)
    t_all, f_all = 0.0, 0.0
    for _ in range(args.steps):
        t, f = oracle_sample_run(ops)
        t_all += t
        f_all += f
    v = f_all / t_all / 1e12
    sample = (f"fp64 oracle, every {stride}th row of each of the 32 sweep GEMMs per step "
              f"({f_all / args.steps / 1e9:.2f} GFLOP per step)")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_all / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": sweep_config(world),
            "api": "the fp64 oracle (oracle_gemm) on a row sample of each sweep GEMM",
            "cpu_baseline": {"value": v, "unit": "TFLOP/s", "cores": oracle.num_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------- single case
def run_case(args):
    """Times one hot-path call on its own (for profiling and sweeps):
    sweep (the 32 sweep GEMMs in one grouped call) | fp8 | mx (the 16 K-major sweep shapes as
    E4M3 / block-scaled E4M3 in one grouped call) | gemm:M,N,K,transA,transB,beta |
    gru[:T,batch,hidden] | gru_rb[:T,batch,hidden] (reset gate before the candidate's
    product) | gru_stack[:L,T,batch,hidden] | gru_stack_rb[:...] | gru_layers[:...] (the
    stack as one call per layer) | dwsep[:N,H,W,Cin,Cout]."""
    import torch
    from paper_1810_09958_gb300 import build, isam, synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    if not os.path.exists(isam.LIB_PATH):
        build.build()
    isam.load()
    kind, _, rest = args.case.partition(":")
    vals = [float(v) for v in rest.split(",")] if rest else []
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    if kind == "gemm":
        M, N, K, tA, tB = (int(v) for v in vals[:5])
        beta = vals[5] if len(vals) > 5 else 0.0
        A = synth.bf16_uniform_torch(11, M * K, dev)
        B = synth.bf16_uniform_torch(12, K * N, dev)
        C = synth.f32_uniform_torch(13, M * N, dev)
        fn = lambda: isam.gemm(M, N, K, tA, tB, 1.0, A, B, beta, C)
        work = {"tflops": gemm_flops(M, N, K) / 1e12, "gb": gemm_bytes(M, N, K, beta != 0) / 1e9,
                "plan": isam.gemm_plan(M, N, K, tA, tB, beta)}
    elif kind == "sweep":
        probs = make_sweep(dev)
        call = isam.GroupedGemm([(p["M"], p["N"], p["K"], p["tA"], 0, 1.0, p["A"], p["B"], 0.0, p["C"])
                                 for p in probs])
        fn = call
        work = {"tflops": sum(p["flops"] for p in probs) / 1e12,
                "gb": sum(p["bytes"] for p in probs) / 1e9}
    elif kind in ("fp8", "mx"):
        # the 16 K-major sweep shapes on E4M3 operands in one grouped call;
        # "mx" adds one E8M0 scale per 32 K elements of each row of A and B
        probs = []
        by = 0
        for (M, K) in SWEEP_MK:
            for N_ in SWEEP_N:
                seed = synth.stream_seed(synth.BASE_SEED, 7, M, K, N_)
                A_ = synth.e4m3_uniform_torch(synth.stream_seed(seed, 1), M * K, dev)
                B_ = synth.e4m3_uniform_torch(synth.stream_seed(seed, 2), N_ * K, dev)
                C_ = torch.empty(M * N_, dtype=torch.float32, device=dev)
                if kind == "mx":
                    SA = torch.full((isam.mx_scale_bytes(M, K),), 127, dtype=torch.uint8, device=dev)
                    SB = torch.full((isam.mx_scale_bytes(N_, K),), 127, dtype=torch.uint8, device=dev)
                    probs.append((M, N_, K, 1.0, A_, SA, B_, SB, 0.0, C_))
                    by += M * K + N_ * K + isam.mx_scale_bytes(M + N_, K) + 4 * M * N_
                else:
                    probs.append((M, N_, K, 1.0, A_, B_, 0.0, C_))
                    by += M * K + N_ * K + 4 * M * N_
        fn = isam.GroupedGemmMxfp8(probs) if kind == "mx" else isam.GroupedGemmFp8(probs)
        work = {"tflops": sum(2.0 * q[0] * q[1] * q[2] for q in probs) / 1e12, "gb": by / 1e9}
    elif kind in ("gru", "gru_rb"):
        T, batch, H = (int(v) for v in vals) if vals else (128, 32, 1024)
        s = H ** -0.5
        x = synth.bf16_normal_torch(21, T * batch * H, dev)
        W = synth.bf16_uniform_torch(22, 3 * H * H, dev, -s, s)
        U = synth.bf16_uniform_torch(23, 3 * H * H, dev, -s, s)
        b = synth.f32_uniform_torch(24, 6 * H, dev, -0.1, 0.1)
        hout = torch.empty(T * batch * H, dtype=torch.float32, device=dev)
        rb = kind == "gru_rb"
        fn = lambda: isam.gru_forward(T, batch, H, x, W, U, b, None, hout, reset_before=rb)
        work = {"tflops": 2.0 * T * batch * 3 * H * 2 * H / 1e12, "timesteps": T}
    elif kind in ("gru_stack", "gru_stack_rb", "gru_layers"):
        L, T, batch, H = (int(v) for v in vals) if vals else (2, 128, 32, 1024)
        s = H ** -0.5
        x = synth.bf16_normal_torch(21, T * batch * H, dev)
        W = synth.bf16_uniform_torch(22, L * 3 * H * H, dev, -s, s)
        U = synth.bf16_uniform_torch(23, L * 3 * H * H, dev, -s, s)
        b = synth.f32_uniform_torch(24, L * 6 * H, dev, -0.1, 0.1)
        hout = torch.empty(L * T * batch * H, dtype=torch.float32, device=dev)
        if kind == "gru_layers":
            # the same stack as one isam_gru_forward call per layer, with a bf16
            # cast of each layer's states (a torch kernel) as the next input
            xs = [x] + [torch.empty(T * batch * H, dtype=torch.bfloat16, device=dev) for _ in range(L - 1)]
            seq = T * batch * H

            def fn():
                for l in range(L):
                    if l > 0:
                        xs[l].copy_(hout[(l - 1) * seq:l * seq])
                    isam.gru_forward(T, batch, H, xs[l], W[l * 3 * H * H:(l + 1) * 3 * H * H],
                                     U[l * 3 * H * H:(l + 1) * 3 * H * H], b[l * 6 * H:(l + 1) * 6 * H],
                                     None, hout[l * seq:(l + 1) * seq])
        else:
            rb = kind == "gru_stack_rb"
            fn = lambda: isam.gru_forward_stack(L, T, batch, H, x, W, U, b, None, hout, reset_before=rb)
        work = {"tflops": L * 2.0 * T * batch * 3 * H * 2 * H / 1e12, "timesteps": T}
    elif kind == "dwsep":
        N, H, W, Cin, Cout = (int(v) for v in vals) if vals else (32, 56, 56, 128, 256)
        x = synth.bf16_normal_torch(31, N * H * W * Cin, dev)
        dw = synth.bf16_uniform_torch(32, 9 * Cin, dev, -1 / 3, 1 / 3)
        pw = synth.bf16_uniform_torch(33, Cin * Cout, dev, -Cin ** -0.5, Cin ** -0.5)
        out = torch.empty(N * H * W * Cout, dtype=torch.float32, device=dev)
        fn = lambda: isam.dwsep_conv(N, H, W, Cin, Cout, x, dw, pw, out)
        work = {"gb": (N * H * W * (2 * Cin + 4 * Cout) + 18 * Cin + 2 * Cin * Cout) / 1e9,
                "tflops": 2.0 * N * H * W * Cin * (9 + Cout) / 1e12}
    else:
        raise SystemExit(f"unknown case {args.case}")
    ms = time_call(fn, reps=args.steps, warmup=args.warmup, flush=flush)
    isam.sync()
    res = {"case": args.case, "ms": round(ms, 5)}
    if "tflops" in work:
        res["tflops_per_s"] = round(work["tflops"] / (ms / 1e3), 2)
    if "gb" in work:
        res["gb_per_s"] = round(work["gb"] / (ms / 1e3), 1)
    if "timesteps" in work:
        res["timesteps_per_s"] = round(work["timesteps"] / (ms / 1e3), 1)
    if "plan" in work:
        res["plan"] = work["plan"]
    print(json.dumps(res), flush=True)
    return 0


# --------------------------------------------------------------------------- main
def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["isam", "reference"], default="isam")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-hot-path", action="store_true")
    ap.add_argument("--case", default=None,
                    help="time one call instead of the benchmark: sweep (grouped) | gemm:M,N,K,tA,tB,beta | "
                         "gru[:T,batch,hidden] | gru_rb[:T,batch,hidden] | dwsep[:N,H,W,Cin,Cout]")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        args.warmup = 3
    if args.case:
        return run_case(args)

    if args.impl == "reference":
        return reference_arm(args)

    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    from paper_1810_09958_gb300 import build, isam
    if not os.path.exists(isam.LIB_PATH):
        build.build()
    isam.load()
    peaks, peaks_src = read_peaks()

    probs = make_sweep(dev)
    torch.cuda.synchronize()
    sampler = ClockSampler(dev.index).start() if rank == 0 else None
    time.sleep(0.3)
    flops_step = sum(p["flops"] for p in probs)
    bytes_step = sum(p["bytes"] for p in probs)

    # value: one isam_gemm_grouped launch per step over the 32 problems.
    kern_ms, window = time_grouped(isam, probs, args.steps, args.warmup)
    total_ms = reduce_max(kern_ms, dev)
    value = whole_job_tflops(flops_step, args.steps, world, total_ms)
    launches = args.steps

    # The same sweep as 32 separate isam_gemm launches per step.
    call_ms, _ = time_sweep(isam, probs, args.steps, args.warmup)
    call_ms = reduce_max(call_ms, dev)
    call_value = whole_job_tflops(flops_step, args.steps, world, call_ms)

    e2e_steps = max(20, args.steps // 20)
    e2e_ms, h2d, d2h = time_e2e(isam, probs, e2e_steps, args.warmup)
    e2e_ms = reduce_max(e2e_ms, dev)
    e2e_value = whole_job_tflops(flops_step, e2e_steps, world, e2e_ms)

    hot, hot_windows = None, {}
    if not args.no_hot_path:
        hot, hot_windows = hot_path_rows(isam, dev, peaks)
        t0 = time.time()
        shape_rows = per_shape_table(isam, dev, peaks)
        shape_rows_f8 = per_shape_table(isam, dev, peaks, fp8=True)
        hot_windows["per_shape"] = (t0, time.time())
    if sampler:
        sampler.stop()
        if hot is not None:
            for name, win in hot_windows.items():
                if name in hot:
                    hot[name]["clocks"] = sampler.summary(*win)
            hot["gru_stack2_h1024_b32_t128"]["per_layer_clocks"] = sampler.summary(
                *hot_windows["gru_stack2_per_layer"])
    del probs
    torch.cuda.empty_cache()

    if rank == 0:
        achieved = bytes_step * args.steps / (kern_ms / 1e3) / 1e9
        call_gbs = bytes_step * args.steps / (call_ms / 1e3) / 1e9
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": sweep_config(world),
            "api": "isam_gemm_grouped: the 32 GEMMs of a step in one call",
            "roofline": {"kernel": "gemm_group_kernel", "bound": "hbm", "achieved": round(achieved, 1),
                         "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": round(achieved / peaks["hbm_gbs"], 4), "traffic": TRAFFIC_PER_STEP,
                         "peak_source": peaks_src,
                         "algorithmic_bytes_per_launch": bytes_step,
                         "launches_per_step": 1,
                         "timing": "one launch per step, replayed from a CUDA graph; duration = "
                                   "timed-region CUDA events on the replay stream / steps"},
            "e2e": {"value": round(e2e_value, 3), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                    "what": "per step: every operand copied in from one pinned host buffer (one copy), isam_gemm_grouped, every result copied out to one pinned host buffer (one copy); two device operand sets, step k+1 inputs copied while step k computes"},
            "gpu_launches": launches,
            "clocks": sampler.summary(*window) if sampler else None,
            "per_call_sweep": {
                "value": round(call_value, 3), "unit": "TFLOP/s",
                "ms_per_step": round(call_ms / args.steps, 5), "achieved_gbs": round(call_gbs, 1),
                "frac_hbm": round(call_gbs / peaks["hbm_gbs"], 4), "launches_per_step": 32,
                "what": "the same 32 GEMMs as 32 isam_gemm calls per step (gemm_tc_kernel), "
                        "graph-replayed; inter-launch gaps included"},
        }
        if hot is not None:
            line["hot_path"] = hot
            line["per_shape"] = {
                "what": "each sweep shape alone through the per-call API, back-to-back calls on "
                        "their own operand sets (>= 256 MB per replay), CUDA-event time per call",
                "clocks": sampler.summary(*hot_windows["per_shape"]) if sampler else None,
                "isam_gemm": shape_rows, "isam_gemm_fp8": shape_rows_f8}
        if not args.no_cpu_baseline and world == 1:
            import oracle
            oracle.build()
            line["cpu_baseline"] = cpu_baseline()
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

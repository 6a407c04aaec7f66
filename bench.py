#!/usr/bin/env python
"""Benchmark of the ESB inference hot path on GB300 (one JSON line on stdout).

Workload (default): a ResNet18-shaped 3x3 convolution layer, NHWC, batch 32,
56x56, 64 -> 64 channels, stride 1, pad 1, weights and activations in
ESB(4,2) (activations post-ReLU, unsigned).  Inputs are seeded synthetic
tensors: X ~ |N(0,1)|, W ~ N(0, sqrt(2/576)) (He init).

One step = one pass of the hot path over one batch, captured as a CUDA
graph:
  esb_project_dda(X)   (DDA statistics and alpha of the batch, then its
                        projection to packed codes, in one launch)
  esb_conv2d_nhwc(Xc, Wc) with the fused epilogue (dequant scale from the two
  device alphas, ReLU, ESB requantisation with the layer's calibrated
  output alpha) -> next layer's packed codes.
The weights are calibrated and projected once at set-up with the same
entry points (esb_calibrate_dda, esb_project), as a deployed layer stores
W already in ESB codes.
Consecutive steps take their input from a rotation of NBATCH seeded
batches whose fp32 activations together exceed the 129 MB L2 (no step
finds its input in L2).  One CUDA graph holds NBATCH consecutive steps (so
kernel boundaries inside it keep their programmatic launch edges); the K
timed steps are K // NBATCH replays of it plus a graph of the remaining
steps, bracketed by CUDA events on the launching stream.  `value` is conv TOPS over the whole step (2 ops per
MAC).  --impl reference times the CPU oracle instead.
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
sys.path.insert(0, ROOT)

METRIC = "ESB GEMM/conv int TOPS and esb_project GB/s, % of GB300 roofline (1 GPU)"
UNIT = "TOPS"

N_, H_, W_, C_, CO_, R_, S_ = 32, 56, 56, 64, 64, 3, 3
STRIDE, PAD = 1, 1
FB, FK = 4, 2
P_ = (H_ + 2 * PAD - R_) // STRIDE + 1
Q_ = (W_ + 2 * PAD - S_) // STRIDE + 1
MACS = N_ * P_ * Q_ * CO_ * R_ * S_ * C_
OPS = 2 * MACS
WORKLOAD = {"workload": "resnet18_conv3x3_56x56_b32_esb42", "n": N_, "h": H_, "w": W_, "c": C_, "cout": CO_,
            "r": R_, "s": S_, "stride": STRIDE, "pad": PAD, "b": FB, "k": FK, "ops_per_step": OPS,
            "l2": "inputs rotated over 6 batches (154 MB of fp32 activations > 129 MB L2), no flush"}
NBATCH = 6


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], "measured"
    return 6800.0, 1900.0, "fallback"


# The sources of each timed kernel and the ncu summary (profiles/) that
# holds its DRAM traffic per launch.
KERNEL_SOURCES = {
    "conv": (("esb_conv_halo.cu", "esb_tc.cuh", "esb_gemm.cu", "esb_common.cuh"), "conv3x3_b32_ncu.txt"),
    "project_dda_x": (("esb_quant.cu", "esb_common.cuh"), "project_dda_b32_ncu.txt"),
}


def _kernel_hash(kind):
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kind][0]:
        h.update(open(os.path.join(ROOT, "paper_2109_03513_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def _traffic_from_profile(kind):
    """DRAM bytes per launch of a kernel from its committed ncu summary, if it
    was taken on the current kernel source; else None."""
    p = os.path.join(ROOT, "profiles", KERNEL_SOURCES[kind][1])
    if not os.path.exists(p):
        return None
    kernel_hash = _kernel_hash(kind)
    kv = {}
    for line in open(p):
        if ":" in line:
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("kernel_source_hash") != kernel_hash:
        return None
    try:
        return float(kv["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    def __init__(self):
        self.proc = None
        self.path = os.path.join("/tmp", f"esb_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self, gpu_index=0):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        with open(self.path) as fh:
            lines = fh.readlines()
        os.unlink(self.path)
        return summarise_clocks(lines, gpu_index)


def summarise_clocks(lines, gpu_index=0):
    """The clocks object of the JSON line from nvidia-smi CSV samples (index,
    clocks.sm, clocks.max.sm, power.draw, reasons.active, hw_slowdown,
    hw_thermal_slowdown, sw_thermal_slowdown, sw_power_cap): median SM clock,
    the maximum, and every throttle reason seen active in any sample."""
    rows = []
    for line in lines:
        parts = [x.strip() for x in line.split(",")]
        if len(parts) >= 9 and parts[0] == str(gpu_index):
            rows.append(parts)
    if not rows:
        return None
    mhz = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
    reasons = set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for r in rows:
        for name, v in zip(names, r[5:9]):
            if v.lower().startswith("active"):
                reasons.add(name)
    return {"sm_mhz": statistics.median(mhz) if mhz else None, "sm_max_mhz": float(rows[0][2]),
            "samples": len(rows), "reasons": sorted(reasons)}


# --------------------------------------------------------------------- GPU arm

def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2109_03513_gb300 import esb, synth
    import __graft_entry__

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0 or world == 1:
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    esb.lib()

    fu, fs = esb.Fmt(FB, FK, False), esb.Fmt(FB, FK, True)
    xs_h = [synth.half_normal((N_ * H_ * W_, C_), seed=1 + rank * NBATCH + i) for i in range(NBATCH)]
    x_h = xs_h[0]
    w_h = synth.he_normal((CO_ * R_ * S_, C_), fan_in=R_ * S_ * C_, seed=2)
    Xs = [t.to(dev) for t in xs_h]
    X = Xs[0]
    Wt = w_h.to(dev)
    ldx = esb.esb_row_words(C_, FB)
    Xcs = [torch.empty((N_ * H_ * W_, ldx), dtype=torch.int32, device=dev) for _ in range(NBATCH)]
    Xc = Xcs[0]
    Wc = torch.empty((CO_ * R_ * S_, ldx), dtype=torch.int32, device=dev)
    M = N_ * P_ * Q_
    Yc = torch.empty((M, esb.esb_row_words(CO_, FB)), dtype=torch.int32, device=dev)
    ax = torch.empty(1, dtype=torch.float32, device=dev)
    aw = torch.empty(1, dtype=torch.float32, device=dev)
    # calibration workspaces: zero-filled once, left zero by every call
    wsx = torch.zeros(esb.esb_calibrate_dda_workspace_bytes(X.numel()), dtype=torch.uint8, device=dev)
    wsw = torch.zeros(esb.esb_calibrate_dda_workspace_bytes(Wt.numel()), dtype=torch.uint8, device=dev)

    # Weights: calibrated and projected once (a deployed layer stores ESB codes).
    # Output alpha of the layer: one untimed calibration pass over the fp32
    # ReLU output of batch 0.
    esb.esb_calibrate_dda(Wt, fs, alpha_out=aw, workspace=wsw)
    esb.esb_project(Wt, fs, alpha=aw, codes=Wc)
    esb.esb_calibrate_dda(X, fu, alpha_out=ax, workspace=wsx)
    esb.esb_project(X, fu, alpha=ax, codes=Xc)
    ep_cal = esb.Epilogue(scale0=1.0, alpha_a_dev=ax, alpha_b_dev=aw, act=esb.ESB_ACT_RELU, alpha_out=1.0,
                          fmt_out=fu)
    _, y32, _ = esb.esb_conv2d_nhwc(Xc, fu, Wc, fs, N_, H_, W_, C_, CO_, R_, S_, STRIDE, PAD, ep=ep_cal,
                                    want_acc=False, want_y=True)
    a_out, _ = esb.esb_calibrate_dda(y32, fu)
    del y32
    alpha_out = float(a_out.item())
    ep = esb.Epilogue(scale0=1.0, alpha_a_dev=ax, alpha_b_dev=aw, act=esb.ESB_ACT_RELU, alpha_out=alpha_out,
                      fmt_out=fu)

    stream = torch.cuda.Stream(device=dev)

    def calls_for(i):
        Xi, Xci = Xs[i], Xcs[i]
        return [
            ("project_dda_x", lambda: esb.esb_project_dda(Xi, fu, alpha_out=ax, workspace=wsx, codes=Xci,
                                                          stream=stream), 1),
            ("conv", lambda: esb.esb_conv2d_nhwc(Xci, fu, Wc, fs, N_, H_, W_, C_, CO_, R_, S_, STRIDE, PAD, ep=ep,
                                                 want_acc=False, out_codes=Yc, stream=stream), 1),
        ]

    calls = calls_for(0)
    launches_per_step = sum(c[2] for c in calls)

    with torch.cuda.stream(stream):
        for i in range(NBATCH):
            for _, fn, _ in calls_for(i):
                fn()
    torch.cuda.synchronize(dev)
    def capture(steps):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(steps):
                for _, fn, _ in calls_for(i):
                    fn()
        return g

    # graph_all: NBATCH consecutive steps (batches 0 .. NBATCH-1); graph_one:
    # the step of batch 0 (end-to-end timing); graph_rem: the first
    # K % NBATCH steps, so that exactly K steps are timed
    graph_all = capture(NBATCH)
    graph_one = capture(1)
    graph_rem = capture(args.steps % NBATCH) if args.steps % NBATCH else None
    torch.cuda.synchronize(dev)

    with torch.cuda.stream(stream):
        for i in range((args.warmup + NBATCH - 1) // NBATCH):
            graph_all.replay()
    torch.cuda.synchronize(dev)

    K = args.steps
    t0e, t1e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler()
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        t0e.record(stream)
        for i in range(K // NBATCH):
            graph_all.replay()
        if graph_rem is not None:
            graph_rem.replay()
        t1e.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ck = clocks.stop(local)
    t_ms = t0e.elapsed_time(t1e)
    assert esb.esb_get_status(stream) == 0
    t_max = t_ms
    if world > 1:
        tt = torch.tensor([t_ms], dtype=torch.float64, device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        t_max = float(tt.item())
    value = world * K * OPS / (t_max * 1e-3) / 1e12

    # Per-kernel durations (same launches, un-graphed, rotating inputs) for the
    # roofline.  A device-side sleep in front of each chain keeps the GPU busy
    # while the host enqueues every launch, so the events see GPU time only.
    reps = max(24, min(240, K // 10))
    per = {name: 0.0 for name, _, _ in calls}
    with torch.cuda.stream(stream):
        for rep in range(reps):
            cl = calls_for(rep % NBATCH)
            evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(cl) + 1)]
            torch.cuda._sleep(2_000_000)
            evs[0].record(stream)
            for j, (_, fn, _) in enumerate(cl):
                fn()
                evs[j + 1].record(stream)
            torch.cuda.synchronize(dev)
            for j, (name, _, _) in enumerate(cl):
                per[name] += evs[j].elapsed_time(evs[j + 1]) / reps

    # End to end through the public API with host buffers: H2D of X, the step,
    # D2H of the output codes, all inside the timed region.
    x_pin = x_h.pin_memory()
    y_pin = torch.empty(Yc.shape, dtype=torch.int32).pin_memory()
    ke = max(10, min(200, K // 10))
    with torch.cuda.stream(stream):
        for i in range(3):
            X.copy_(x_pin, non_blocking=True)
            graph_one.replay()
            y_pin.copy_(Yc, non_blocking=True)
        torch.cuda.synchronize(dev)
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(ke):
            X.copy_(x_pin, non_blocking=True)
            graph_one.replay()
            y_pin.copy_(Yc, non_blocking=True)
        a1.record(stream)
        torch.cuda.synchronize(dev)
    e2e_ms = a0.elapsed_time(a1) / ke
    e2e_value = world * OPS / (e2e_ms * 1e-3) / 1e12
    if world > 1:
        tt = torch.tensor([e2e_ms], dtype=torch.float64, device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        e2e_value = world * OPS / (float(tt.item()) * 1e-3) / 1e12

    hbm, bf16, src = _peaks()
    n_x, n_w = X.numel(), Wt.numel()
    algo = {  # algorithmic bytes / ops per launch
        # one HBM read of x (the second pass reads it from L2) + the code words written
        "project_dda_x": ("hbm", 4.0 * n_x + 4.0 * Xc.numel()),
        "conv": ("tensor", float(OPS)),
    }
    dominant = max(per, key=per.get)
    bound, amount = algo[dominant]
    t_k = per[dominant] * 1e-3
    khash = {kind: _kernel_hash(kind) for kind in KERNEL_SOURCES}
    if bound == "tensor":
        achieved = amount / t_k / 1e12
        peak = 2.0 * bf16
        roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "kernel": dominant,
                "peak_note": f"fp8 dense = {src} bf16 burst {bf16} x nominal fp8:bf16 ratio 2",
                "traffic": _traffic_from_profile(dominant)}
    else:
        achieved = amount / t_k / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "kernel": dominant, "peak_note": f"{src} HBM copy", "traffic": _traffic_from_profile(dominant)}
    kernels = {}
    for name, (b, amt) in algo.items():
        t = per[name] * 1e-3
        if b == "tensor":
            kernels[name] = {"us": per[name] * 1e3, "TFLOP/s": amt / t / 1e12, "frac": amt / t / 1e12 / (2.0 * bf16)}
        else:
            kernels[name] = {"us": per[name] * 1e3, "GB/s": amt / t / 1e9, "frac": amt / t / 1e9 / hbm}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": args.warmup,
        "ms_per_step": t_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3", "data": "synthetic (seeded |N(0,1)| activations, He-init N(0,sqrt(2/576)) weights)",
        "config": dict(WORKLOAD, parallelism="replicas" if world > 1 else "single"),
        "roofline": roof, "kernels": kernels,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(x_pin.numel() * 4),
                "d2h_bytes_per_step": int(y_pin.numel() * 4), "ms_per_step": e2e_ms},
        "gpu_launches": launches_per_step * K,
        "clocks": ck, "kernel_source_hash": khash,
    }
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ----------------------------------------------------------- CPU oracle arm

class OracleSample:
    """The benchmark step by the CPU oracle on a bounded sample of the
    workload: DDA calibration and projection of the input rows that the
    sampled output rows read (all of X when the sample is the whole batch),
    then conv + epilogue of those output rows (image-major).  The weights are
    calibrated and projected once, as the GPU arm does at set-up.  The work
    of a step is proportional to its rows, so a step can be made as short as
    one output row.  run() returns the conv ops it performed."""

    def __init__(self, pool):
        import numpy as np

        import oracle as o
        from paper_2109_03513_gb300 import synth

        o.build()
        self.np, self.o, self.pool = np, o, pool
        self.x = synth.half_normal((N_ * H_ * W_, C_), seed=1).numpy()
        w = synth.he_normal((CO_ * R_ * S_, C_), fan_in=R_ * S_ * C_, seed=2).numpy()
        self.ldx = (-(-C_ // (32 // FB)) + 3) // 4 * 4
        self.aw, _ = o.calibrate(w, FB, FK, signed=True)
        self.Wc = o.project_packed(w, self.aw, FB, FK, True, ld_words=self.ldx).reshape(CO_, R_, S_, self.ldx)
        self.zero_row = o.pack(np.full((1, C_), o.zero_code(FB, FK), np.uint32), FB, FK, ld_words=self.ldx)[0]

    def run(self, rows):
        np, o = self.np, self.o
        units = [(i // P_, i % P_) for i in range(rows)]
        need = sorted({(n, p * STRIDE - PAD + r) for n, p in units for r in range(R_)
                       if 0 <= p * STRIDE - PAD + r < H_})
        sample = np.concatenate([self.x[(n * H_ + h) * W_:(n * H_ + h + 1) * W_] for n, h in need])
        ax, _ = o.calibrate(sample, FB, FK, signed=False)
        imgs = {n: np.tile(self.zero_row, (1, H_, W_, 1)) for n in sorted({n for n, _ in need})}
        chunks = [need[i:i + 64] for i in range(0, len(need), 64)]

        def proj(ch):
            for n, h in ch:
                src = self.x[(n * H_ + h) * W_:(n * H_ + h + 1) * W_]
                imgs[n][0, h] = o.project_packed(src, ax, FB, FK, False, ld_words=self.ldx)

        list(self.pool.map(proj, chunks))
        scale = np.float32(np.float32(ax) * np.float32(self.aw)) * np.float32(2.0 ** -(2 * FK))

        # few rows: split each row's output channels over the threads too
        split = 8 if rows < self.pool._max_workers else 1
        cw = CO_ // split

        def one(u):
            (n, p), g = u
            acc = o.conv2d_rows_i64(imgs[n], (FB, FK), self.Wc[g * cw:(g + 1) * cw], (FB, FK), 1, H_, W_, C_, cw,
                                    R_, S_, STRIDE, PAD, p, p + 1)
            o.epilogue(acc.reshape(-1, cw), np.full(cw, scale, np.float32), np.zeros(cw, np.float32), 1,
                       0.25, (FB, FK, False))
            return cw

        done = sum(self.pool.map(one, [(u, g) for u in units for g in range(split)]))
        return 2 * done * Q_ * R_ * S_ * C_

    def rows_for_budget(self, seconds):
        """Rows per step so that a step takes about `seconds` (at least one
        row): a + b * rows fitted from two timed runs."""
        import time as _t
        cores = self.pool._max_workers
        r2 = min(N_ * P_, 4 * cores)
        t0 = _t.perf_counter()
        self.run(1)
        t1 = _t.perf_counter()
        self.run(r2)
        t2 = _t.perf_counter()
        a, ta2 = t1 - t0, t2 - t1
        b = max((ta2 - a) / max(r2 - 1, 1), 1e-6)
        return int(max(1, min(N_ * P_, 1 + (seconds - a) / b)))


def _cores():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)


def cpu_baseline(budget_s=12.0):
    from concurrent.futures import ThreadPoolExecutor

    cores = _cores()
    with ThreadPoolExecutor(max_workers=cores) as pool:
        smp = OracleSample(pool)
        rows = smp.rows_for_budget(budget_s)
        t0 = time.perf_counter()
        ops = smp.run(rows)
        dt = time.perf_counter() - t0
    return {"value": ops / dt / 1e12, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"DDA calibration and projection of the input rows read by {rows} of the {N_ * P_} "
                      f"output rows of X ({N_}x{H_}x{W_}x{C_}; all of X when all rows), conv + epilogue of those "
                      f"rows ({ops / 1e9:.3f} GOP; weights projected once at set-up); {dt:.2f} s wall",
            "seconds": dt}


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from concurrent.futures import ThreadPoolExecutor

    cores = _cores()
    times = []
    ops = 0
    with ThreadPoolExecutor(max_workers=cores) as pool:
        smp = OracleSample(pool)
        budget = 120.0 / (args.steps + args.warmup)           # whole run within a few minutes
        rows = smp.rows_for_budget(budget)
        for i in range(args.warmup + args.steps):
            t0 = time.perf_counter()
            ops = smp.run(rows)
            dt = time.perf_counter() - t0
            if i >= args.warmup:
                times.append(dt)
    total = sum(times)
    value = len(times) * ops / total / 1e12
    sample = (f"per step: DDA calibration and projection of the input rows read by {rows} of the {N_ * P_} "
              f"output rows, conv + epilogue of those rows ({ops / 1e9:.3f} GOP; weights projected once at set-up)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
            "data": "synthetic", "config": dict(WORKLOAD, parallelism="cpu oracle"),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_sweep(args):
    """The sweeps of the large-operand workloads, one JSON line: esb_gemm_tiled
    on square M=N=K in {1024, 4096, 8192, 16384} at ESB (4,2) and (6,3)
    (unsigned A, signed B, codes out), and esb_project on 2^28 fp32 values
    drawn N(0,1), Laplace(0,1) and |N(0,1)| for every b in 3..6, k in 1..b-1
    with the tensor's DDA alpha (`--sweeps gemm` / `--sweeps project` run
    one part).  Each point: CUDA events over
    repeated calls after 3 warm-ups (operands larger than L2 from 4096 up;
    the projection reads 1 GiB per call)."""
    import torch

    from paper_2109_03513_gb300 import esb, synth
    import __graft_entry__

    __graft_entry__.build()
    dev = torch.device("cuda")
    hbm, bf16, _ = _peaks()
    fp8 = 2.0 * bf16
    st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timeit(f, reps):
        for _ in range(3):
            f()
        torch.cuda.synchronize()
        st.record()
        for _ in range(reps):
            f()
        en.record()
        torch.cuda.synchronize()
        return st.elapsed_time(en) / reps * 1e3

    out = []
    g = torch.Generator().manual_seed(0)
    if args.sweeps in ("all", "gemm"):
        # the small GEMM of the first configuration: 64 x 64 x 576 at (4,2)
        # (one 3x3x64 conv tile), codes out; a CUDA graph of 200 calls, so the
        # figure is the device time per call without launch gaps
        M_, N_, K_ = 64, 64, 576
        fu, fs = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)
        ld = esb.esb_row_words(K_, 4)
        A = torch.randint(-2 ** 31, 2 ** 31 - 1, (M_, ld), generator=g, dtype=torch.int64).to(torch.int32).to(dev)
        B = torch.randint(-2 ** 31, 2 ** 31 - 1, (N_, ld), generator=g, dtype=torch.int64).to(torch.int32).to(dev)
        A &= 0x77777777                                   # unsigned A: sign bits cleared
        oc = torch.empty((M_, esb.esb_row_words(N_, 4)), dtype=torch.int32, device=dev)
        ep = esb.Epilogue(scale0=1e-3, act=esb.ESB_ACT_RELU, alpha_out=0.3, fmt_out=esb.Fmt(4, 2, False))
        call = lambda: esb.esb_gemm(A, fu, B, fs, K_, ep=ep, want_acc=False, out_codes=oc)
        s_ = torch.cuda.Stream()
        s_.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s_):
            for _ in range(3):
                call()
        torch.cuda.current_stream().wait_stream(s_)
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            for _ in range(200):
                call()
        us = timeit(gr.replay, 10) / 200
        tf = 2.0 * M_ * N_ * K_ / us / 1e6
        out.append({"gemm": [M_, N_, K_], "fmt": [4, 2], "us": round(us, 3), "TFLOP/s": round(tf, 2),
                    "frac_fp8": round(tf / fp8, 5), "note": "CUDA graph of 200 calls, device time per call",
                    "status": esb.esb_get_status()})
        del A, B, oc
    for b, k in ([(4, 2), (6, 3)] if args.sweeps in ("all", "gemm") else []):
        fu, fs = esb.Fmt(b, k, False), esb.Fmt(b, k, True)
        for n in [1024, 4096, 8192, 16384]:
            ld = esb.esb_row_words(n, b)
            # uniformly drawn codes (sign bit cleared for the unsigned A)
            ca = torch.randint(0, 2 ** b, (n, n), generator=g, dtype=torch.int64)
            cb = torch.randint(0, 2 ** b, (n, n), generator=g, dtype=torch.int64)
            ca &= (1 << (b - 1)) - 1
            cpw = 32 // b

            def pack(c):
                c = torch.nn.functional.pad(c, (0, ld * cpw - n)).reshape(n, ld, cpw)
                sh = torch.arange(cpw, dtype=torch.int64) * b
                return ((c << sh).sum(-1) & 0xffffffff).to(torch.int64).to(torch.int32)

            A, B = pack(ca).to(dev), pack(cb).to(dev)
            del ca, cb
            ep = esb.Epilogue(scale0=1e-4, act=esb.ESB_ACT_RELU, alpha_out=0.3, fmt_out=esb.Fmt(4, 2, False))
            oc = torch.empty((n, esb.esb_row_words(n, 4)), dtype=torch.int32, device=dev)
            ws = torch.empty(esb.esb_gemm_tiled_workspace_bytes(n, n, n), dtype=torch.uint8, device=dev)
            f = lambda: esb.esb_gemm(A, fu, B, fs, n, ep=ep, want_acc=False, want_codes=True, out_codes=oc,
                                     workspace=ws)
            reps = max(3, min(200, int(1e11 / (2.0 * n ** 3))))
            us = timeit(f, reps)
            tf = 2.0 * n ** 3 / us / 1e6
            out.append({"gemm": [n, n, n], "fmt": [b, k], "us": round(us, 2), "TFLOP/s": round(tf, 1),
                        "frac_fp8": round(tf / fp8, 3), "status": esb.esb_get_status()})
            del A, B, oc, ws
            torch.cuda.empty_cache()
    # esb_project on 2^28 values of each configured distribution (N(0,1),
    # Laplace(0,1) and |N(0,1)|, seeds 0/1/2), every b in 3..6 and k in
    # 1..b-1, the half-normal data in the unsigned format, alpha = the DDA
    # alpha of that tensor (esb_calibrate_dda, not timed)
    for di, dist in enumerate(["normal", "laplace", "half_normal"] if args.sweeps in ("all", "project") else []):
        x = synth.distribution(dist, (1 << 28,), seed=di).to(dev)
        signed = dist != "half_normal"
        for b in range(3, 7):
            for k in range(1, b):
                f = esb.Fmt(b, k, signed)
                a, _ = esb.esb_calibrate_dda(x, f)
                codes = torch.empty((1, esb.esb_row_words(1 << 28, b)), dtype=torch.int32, device=dev)
                us = timeit(lambda: esb.esb_project(x, f, alpha=a, codes=codes), 20)
                byt = (1 << 28) * (4 + 4 / (32 // b))
                out.append({"project": 1 << 28, "dist": dist, "fmt": [b, k, int(signed)], "alpha": float(a.item()),
                            "us": round(us, 1), "GB/s": round(byt / us / 1e3, 1),
                            "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
                del codes
        del x
        torch.cuda.empty_cache()
    if args.sweeps in ("all", "cc"):
        out += _cc_sweep(esb, torch, timeit, hbm)
    print(json.dumps({"workload": "sweeps (esb_gemm_tiled M=N=K, esb_project 2^28, depthwise conv and pooling)",
                      "peaks": {
        "hbm_gbs": hbm, "fp8_tflops": fp8, "note": "measured HBM copy; fp8 = 2 x measured bf16 burst"},
        "results": out}))


def _cc_sweep(esb, torch, timeit, hbm):
    """The CUDA-core kernels at batch 64: MobileNetV2's depthwise 3x3 layers
    (fused scale, bias, ReLU6 and requantisation, codes out), the ResNet18
    stem max pool 112 -> 56 and the global average pools of ResNet18 (7x7x512)
    and MobileNetV2 (7x7x1280), all ESB(4,2).  Algorithmic bytes = input
    codes + output codes (+ weights, scale and bias).  Each point is a CUDA
    graph of one call per input copy (over 3 x L2 of copies in total, so
    inputs come from HBM), replayed; the figure is device time per call,
    without host launch gaps.  Codes are uniformly drawn words (timing only)."""
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(0)
    fx, fw = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)
    n = 64
    span = 3 * 129 * 10 ** 6

    def copies(rows, ld, unsigned):
        nbytes = rows * ld * 4
        nx = max(3, min(256, -(-span // nbytes)))
        c = torch.randint(0, 2 ** 32, (nx * rows, ld), generator=g, device=dev, dtype=torch.int64).to(torch.int32)
        if unsigned:
            c &= 0x77777777
        return [c[i * rows:(i + 1) * rows] for i in range(nx)], nbytes

    def graphed(calls, reps=5):
        s_ = torch.cuda.Stream()
        s_.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s_):
            for f in calls[:3]:
                f()
        torch.cuda.current_stream().wait_stream(s_)
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            for f in calls:
                f()
        return timeit(gr.replay, reps) / len(calls)

    res = []
    for h, c, stride in [(112, 32, 1), (112, 96, 2), (56, 144, 1), (56, 144, 2), (28, 192, 1), (14, 384, 1),
                         (14, 576, 1), (7, 960, 1)]:
        ld = esb.esb_row_words(c, 4)
        P = (h + 2 - 3) // stride + 1
        Xs, xb = copies(n * h * h, ld, True)
        W, _ = copies(9, ld, False)
        W = W[0]
        scale = torch.full((c,), 1e-3, dtype=torch.float32, device=dev)
        bias = torch.zeros((c,), dtype=torch.float32, device=dev)
        ep = esb.Epilogue(scale=scale, bias=bias, act=esb.ESB_ACT_RELU6, alpha_out=0.29, fmt_out=fx)
        oc = torch.empty((n * P * P, ld), dtype=torch.int32, device=dev)

        def dw(X):
            return lambda: esb.esb_conv2d_nhwc(X, fx, W, fw, n, h, h, c, c, 3, 3, stride, 1, groups=c, ep=ep,
                                               want_acc=False, want_codes=True, out_codes=oc)

        us = graphed([dw(X) for X in Xs])
        byt = xb + oc.numel() * 4 + W.numel() * 4 + 8 * c
        res.append({"dwconv": [n, h, h, c, stride], "fmt": [4, 2], "us": round(us, 2),
                    "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
        del Xs, oc
    Xs, xb = copies(n * 112 * 112, 8, True)
    Y = torch.empty((n * 56 * 56, 8), dtype=torch.int32, device=dev)

    def mp(X):
        return lambda: esb.esb_maxpool_nhwc(X, fx, n, 112, 112, 64, 3, 2, 1, out=Y)

    us = graphed([mp(X) for X in Xs])
    byt = xb + Y.numel() * 4
    res.append({"maxpool": [n, 112, 112, 64, 3, 2], "fmt": [4, 2], "us": round(us, 2),
                "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
    del Xs, Y
    for c in (512, 1280):
        ld = esb.esb_row_words(c, 4)
        Xs, xb = copies(n * 49, ld, True)

        def ap(X):
            return lambda: esb.esb_avgpool_nhwc(X, fx, n, 49, c, 1.0 / 49, 0.5, fx)

        us = graphed([ap(X) for X in Xs], reps=20)
        byt = xb + n * ld * 4
        res.append({"avgpool": [n, 7, 7, c], "fmt": [4, 2], "us": round(us, 2),
                    "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
        del Xs
    res.append({"cc_status": esb.esb_get_status()})
    return res


# ------------------------------------------------------ network workloads

NET_BATCH = {"resnet18": 64, "mobilenetv2": 64, "alexnet_fc": 256}
NET_FMTS = {"resnet18": [(3, 1), (4, 2), (5, 2), (6, 3)], "mobilenetv2": [(4, 2)], "alexnet_fc": [(4, 2)]}


class OAct:
    """An activation of the oracle's forward: packed codes on the host."""

    def __init__(self, np_codes, f, a, n, h, w, c):
        self.np, self.f, self.a, self.n, self.h, self.w, self.c = np_codes, f, a, n, h, w, c


class OracleRunner:
    """The oracle's forward of a network, with the weights, alphas and
    formats of a calibrated libesb Runner (same call sequence): conv layers
    split their output rows over host threads (oracle_conv2d_rows_i64)."""

    def __init__(self, rn, pool):
        self.rn, self.pool, self.idx = rn, pool, 0

    def _p(self):
        p = self.rn.params[self.idx]
        self.idx += 1
        return p

    def input(self, x, n, h, w, c):
        import numpy as np
        import oracle as o
        p = self._p()
        f = (self.rn.b, self.rn.k, True)
        codes = o.project_packed(np.ascontiguousarray(x.reshape(-1, c)), p["a"], *f)
        return OAct(codes, f, p["a"], n, h, w, c)

    def conv(self, x, cout, r, s, stride, pad, act=1, res=None, groups=1):
        import numpy as np
        import oracle as o
        from paper_2109_03513_gb300 import esb
        p = self._p()
        dw = groups == x.c and x.c > 1
        W = p["W_np"]
        fw = (self.rn.b, self.rn.k)
        P, Q = esb.conv_out_hw(x.h, x.w, r, s, stride, pad)
        ldx = x.np.shape[1]
        X4 = x.np.reshape(x.n, x.h, x.w, ldx)
        if dw:
            acc = o.dwconv_i64(X4, x.f[:2], W.reshape(r, s, -1), fw, x.n, x.h, x.w, x.c, r, s,
                               stride, pad).reshape(-1, cout)
        else:
            chunks = [(i * P // 16, (i + 1) * P // 16) for i in range(16) if (i + 1) * P // 16 > i * P // 16]
            parts = list(self.pool.map(lambda pr: o.conv2d_rows_i64(X4, x.f[:2], W.reshape(cout, r, s, -1), fw,
                                                                    x.n, x.h, x.w, x.c, cout, r, s,
                                                                    stride, pad, pr[0], pr[1]), chunks))
            acc = np.concatenate(parts, axis=1).reshape(-1, cout)
        signed_out = act == 0
        fo = (self.rn.b, self.rn.k, signed_out)
        s0 = esb.esb_dequant_scale(x.a, esb.Fmt(*x.f), p["aw"], esb.Fmt(self.rn.b, self.rn.k, True))
        res_img, res_scale = None, 0.0
        if res is not None:
            lut = np.array([o.image(v, res.f[0], res.f[1]) for v in range(2 ** res.f[0])], np.int64)
            res_img = lut[o.unpack(res.np, cout, res.f[0])]
            res_scale = esb.esb_dequant_scale(res.a, esb.Fmt(*res.f), 1.0, esb.Fmt(8, 0))
        _, co = o.epilogue(acc, np.full(cout, s0, np.float32), np.zeros(cout, np.float32), act, p["a_out"], fo,
                           res_images=res_img, res_scale=res_scale)
        return OAct(o.pack(co, fo[0], fo[1], ld_words=esb.esb_row_words(cout, fo[0])), fo, p["a_out"], x.n, P, Q, cout)

    def maxpool(self, x, win=3, stride=2, pad=1):
        import oracle as o
        from paper_2109_03513_gb300 import esb
        self._p()
        P, Q = esb.conv_out_hw(x.h, x.w, win, win, stride, pad)
        Y = o.maxpool_codes(x.np.reshape(x.n, x.h, x.w, -1), x.f[0], x.f[1], x.n, x.h, x.w,
                            x.c, win, stride, pad, ld_out=x.np.shape[1]).reshape(x.n * P * Q, -1)
        return OAct(Y, x.f, x.a, x.n, P, Q, x.c)

    def avgpool(self, x):
        import numpy as np
        import oracle as o
        from paper_2109_03513_gb300 import esb
        p = self._p()
        hw = x.h * x.w
        scale = esb.esb_dequant_scale(x.a, esb.Fmt(*x.f), 1.0 / hw, esb.Fmt(8, 0))
        sums = o.avgpool_sum_i64(x.np.reshape(x.n, hw, -1), x.f[0], x.f[1], x.n, hw, x.c)
        y = (np.float32(scale) * sums.astype(np.float32)).astype(np.float32)
        codes = o.pack(o.project_codes(y, p["a_out"], *x.f), x.f[0], x.f[1],
                       ld_words=esb.esb_row_words(x.c, x.f[0]))
        return OAct(codes, x.f, p["a_out"], x.n, 1, 1, x.c)

    def fc(self, x, nout, act=0, workspace=False):
        import numpy as np
        import oracle as o
        from paper_2109_03513_gb300 import esb
        p = self._p()
        fw = (self.rn.b, self.rn.k)
        acc = o.gemm_i64(x.np, x.f[:2], p["W_np"], fw, x.n, nout, x.c)
        fo = (self.rn.b, self.rn.k, act == 0)
        s0 = esb.esb_dequant_scale(x.a, esb.Fmt(*x.f), p["aw"], esb.Fmt(self.rn.b, self.rn.k, True))
        _, co = o.epilogue(acc, np.full(nout, s0, np.float32), np.zeros(nout, np.float32), act, p["a_out"], fo)
        return OAct(o.pack(co, fo[0], fo[1], ld_words=esb.esb_row_words(nout, fo[0])), fo, p["a_out"], x.n, 1, 1, nout)


def run_network(args, name):
    """One JSON line per (b, k): images/s of the whole forward (a CUDA graph
    of every layer's launches), per-layer TOPS, the end-to-end number with
    the input images copied in and the logits' codes copied out, and the
    oracle's forward of a sample of the batch on the host cores."""
    from concurrent.futures import ThreadPoolExecutor

    import numpy as np
    import torch

    import __graft_entry__
    from paper_2109_03513_gb300 import esb, netrun, synth

    __graft_entry__.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    fn, (h, w, c) = netrun.NETWORKS[name]
    batch = NET_BATCH[name]
    fmts = NET_FMTS[name] if not args.bk else [tuple(int(v) for v in t.split(",")) for t in args.bk]
    hbm, bf16, src = _peaks()
    for b, k in fmts:
        rn = netrun.Runner(b, k, seed=1000 * b + k, device=dev)
        x_cal = synth.normal((batch * h * w, c), seed=1).to(dev)
        x = synth.normal((batch * h * w, c), seed=2).to(dev)
        rn.begin("calibrate")
        fn(rn, x_cal, batch)
        torch.cuda.synchronize()
        del x_cal
        launches = 0
        stream = torch.cuda.Stream(device=dev)
        with torch.cuda.stream(stream):
            rn.begin("infer")
            t_host = time.perf_counter()
            fn(rn, x, batch)
            t_host = time.perf_counter() - t_host         # host time to enqueue one eager pass
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                rn.begin("infer")
                out = fn(rn, x, batch)
            for _ in range(max(args.warmup, 3)):
                g.replay()
            torch.cuda.synchronize()
            K = max(1, min(args.steps, 200))
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            clocks = ClockSampler()
            clocks.start()
            time.sleep(0.2)
            e0.record(stream)
            for _ in range(K):
                g.replay()
            e1.record(stream)
            torch.cuda.synchronize()
            ck = clocks.stop(0)
            t_fwd = e0.elapsed_time(e1) / K * 1e-3
            # per-layer device times: one eager pass queued behind a device sleep
            # that outlasts its host enqueue time (3x margin at up to 2.1 GHz), so
            # that every layer is queued before the device reaches it
            rn.marks = []
            torch.cuda._sleep(int(min(2e9, max(5e6, 3.0 * t_host * 2.1e9))))
            m0 = torch.cuda.Event(enable_timing=True)
            m0.record(stream)
            rn.begin("infer")
            fn(rn, x, batch)
            torch.cuda.synchronize()
            marks, rn.marks = [m0] + rn.marks, None
            layer_us = [marks[i].elapsed_time(marks[i + 1]) * 1e3 for i in range(len(marks) - 1)]
            # end to end: pinned host images in, the logits' codes out
            x_pin = x.cpu().pin_memory()
            o_pin = torch.empty(out.codes.shape, dtype=torch.int32).pin_memory()
            ke = max(3, min(20, K))
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            for _ in range(ke):
                x.copy_(x_pin, non_blocking=True)
                g.replay()
                o_pin.copy_(out.codes, non_blocking=True)
            a1.record(stream)
            torch.cuda.synchronize()
            t_e2e = a0.elapsed_time(a1) / ke * 1e-3
        assert esb.esb_get_status(stream) == 0
        macs = sum(li.macs for li in rn.info)
        layers = []
        for li, us in zip(rn.info, layer_us[1:]):
            d = {"kind": li.kind, "shape": li.shape, "us": round(us, 2)}
            if li.macs:
                d["TOPS"] = round(2 * li.macs / (us * 1e-6) / 1e12, 1)
            layers.append(d)
        dense = [(li, us) for li, us in zip(rn.info, layer_us[1:]) if li.kind in ("conv", "fc")]
        top = max(dense, key=lambda t: t[1])
        peak = 2.0 * bf16
        top_tops = 2 * top[0].macs / (top[1] * 1e-6) / 1e12
        line = {
            "metric": METRIC, "value": batch / t_fwd, "unit": "images/s", "n_gpus": 1, "steps": K,
            "warmup": max(args.warmup, 3), "ms_per_step": t_fwd * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "e4m3",
            "data": "synthetic (seeded N(0,1) images, He-init weights, one calibration batch then a timed batch)",
            "config": {"workload": f"{name}_b{batch}_esb{b}{k}", "batch": batch, "b": b, "k": k,
                       "gop_per_forward": round(2 * macs / 1e9, 2),
                       "l2": "weights and activations stay in L2 across replays (a deployed model's steady state)",
                       "parallelism": "single"},
            "TOPS_forward": round(2 * macs / t_fwd / 1e12, 1),
            "roofline": {"bound": "tensor", "kernel": f"{top[0].kind} {top[0].shape}", "achieved": round(top_tops, 1),
                         "peak": peak, "unit": "TFLOP/s", "frac": round(top_tops / peak, 4),
                         "peak_note": f"fp8 dense = {src} bf16 burst {bf16} x nominal fp8:bf16 ratio 2",
                         "traffic": None},
            "layers": layers,
            "e2e": {"value": batch / t_e2e, "unit": "images/s", "h2d_bytes_per_step": int(x_pin.numel() * 4),
                    "d2h_bytes_per_step": int(o_pin.numel() * 4), "ms_per_step": t_e2e * 1e3},
            "gpu_launches": None, "clocks": ck,
        }
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = network_cpu_baseline(rn, fn, x, name, batch, h, w, c)
        print(json.dumps(line), flush=True)
        del g, rn, x


def network_cpu_baseline(rn, fn, x, name, batch, h, w, c):
    """The oracle's forward of one image (all 1000 classes; conv rows over
    the host threads) with the calibrated weights and alphas."""
    from concurrent.futures import ThreadPoolExecutor

    n1 = 8 if name == "alexnet_fc" else 1
    for p in rn.params:
        if "W" in p:
            p["W_np"] = p["W"].cpu().numpy().view("uint32")
    xs = x[: n1 * h * w].cpu().numpy()
    cores = _cores()
    with ThreadPoolExecutor(cores) as pool:
        orn = OracleRunner(rn, pool)
        t0 = time.time()
        fn(orn, xs, n1)
        dt = time.time() - t0
    return {"value": n1 / dt, "unit": "images/s", "cores": cores, "kind": "oracle",
            "sample": f"{n1} of the {batch} images of the timed batch through every layer ({dt:.1f} s wall)"}


def run_peaks(args):
    """Measured tensor-pipe peaks (the tcgen05 f8f6f4 rate the contraction's
    roofline divides by, and the legacy mma.sync s8 rate), one JSON line."""
    import torch

    import __graft_entry__
    from paper_2109_03513_gb300 import esb

    __graft_entry__.build()
    torch.cuda.set_device(0)
    out = {"peaks": {}}
    clocks = ClockSampler()
    clocks.start()
    time.sleep(0.2)
    for name, kind, iters in [("tcgen05_f8f6f4_e4m3", esb.ESB_PEAK_TCGEN05_F8F6F4, 20000),
                              ("mma_sync_s8", esb.ESB_PEAK_MMA_SYNC_S8, 20000)]:
        for _ in range(3):
            esb.esb_peak_launch(kind, iters)
        torch.cuda.synchronize()
        best = 0.0
        for _ in range(10):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            ops = esb.esb_peak_launch(kind, iters)
            e1.record()
            torch.cuda.synchronize()
            best = max(best, ops / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        out["peaks"][name] = {"TFLOP/s" if kind == 0 else "TOPS": round(best, 1)}
    out["clocks"] = clocks.stop(0)
    out["status"] = esb.esb_get_status()
    hbm, bf16, src = _peaks()
    out["bf16_burst_" + src] = bf16
    print(json.dumps(out), flush=True)


def run_cc_profile(args):
    """A few launches of each CUDA-core kernel, untimed: the target of an ncu
    capture (`-k regex:"dwconv3_b4h|maxpool_b4u|avgpool_kernel"`).  Depthwise
    3x3 112x112x32 at batch 32 (per-channel scale and bias, ReLU6, codes
    out), the ResNet18 stem max pool at batch 32 and the 7x7x1280 global
    average pool at batch 64, ESB(4,2), four rounds."""
    import torch

    from paper_2109_03513_gb300 import esb
    import __graft_entry__

    __graft_entry__.build()
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev).manual_seed(0)
    fx, fw = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)

    def words(rows, ld, unsigned=True):
        c = torch.randint(0, 2 ** 32, (rows, ld), generator=g, device=dev, dtype=torch.int64).to(torch.int32)
        return c & 0x77777777 if unsigned else c

    n, h, c = 32, 112, 32
    ld = esb.esb_row_words(c, 4)
    X, W = words(n * h * h, ld), words(9, ld, False)
    ep = esb.Epilogue(scale=torch.full((c,), 1e-3, device=dev), bias=torch.zeros((c,), device=dev),
                      act=esb.ESB_ACT_RELU6, alpha_out=0.29, fmt_out=fx)
    oc = torch.empty((n * h * h, ld), dtype=torch.int32, device=dev)
    Xm, Y = words(n * 112 * 112, 8), torch.empty((n * 56 * 56, 8), dtype=torch.int32, device=dev)
    Xa = words(64 * 49, esb.esb_row_words(1280, 4))
    for _ in range(4):
        esb.esb_conv2d_nhwc(X, fx, W, fw, n, h, h, c, c, 3, 3, 1, 1, groups=c, ep=ep, want_acc=False,
                            want_codes=True, out_codes=oc)
        esb.esb_maxpool_nhwc(Xm, fx, n, 112, 112, 64, 3, 2, 1, out=Y)
        esb.esb_avgpool_nhwc(Xa, fx, 64, 49, 1280, 1.0 / 49, 0.5, fx)
    torch.cuda.synchronize()
    st = esb.esb_get_status()
    print(json.dumps({"cc_profile": "done", "status": st}), flush=True)
    if st != 0:
        raise SystemExit(1)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweeps", nargs="?", const="all", choices=["all", "gemm", "project", "cc"],
                    help="the sweeps instead of the step (all, or only the GEMM, projection or CUDA-core part)")
    ap.add_argument("--workload", default="conv3x3", choices=["conv3x3", "resnet18", "mobilenetv2", "alexnet_fc"],
                    help="conv3x3: the benchmark step (default); the others: whole-network forwards")
    ap.add_argument("--bk", nargs="*", help="formats b,k of a network workload (default: its configuration's)")
    ap.add_argument("--peaks", action="store_true", help="measure the tensor-pipe peaks instead")
    ap.add_argument("--cc-profile", action="store_true",
                    help="a few untimed launches of the CUDA-core kernels (an ncu capture target)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.cc_profile:
        run_cc_profile(args)
    elif args.peaks:
        run_peaks(args)
    elif args.workload != "conv3x3" and args.impl == "ours":
        run_network(args, args.workload)
    elif args.sweeps:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()

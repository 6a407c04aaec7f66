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
    N(0,1) for every b in 3..6, k in 1..b-1 (`--sweeps gemm` / `--sweeps
    project` run one half).  Each point: CUDA events over
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
    x = synth.normal((1 << 28,), seed=0).to(dev) if args.sweeps in ("all", "project") else None
    for b in (range(3, 7) if args.sweeps in ("all", "project") else []):
        for k in range(1, b):
            f = esb.Fmt(b, k, True)
            codes = torch.empty((1, esb.esb_row_words(1 << 28, b)), dtype=torch.int32, device=dev)
            us = timeit(lambda: esb.esb_project(x, f, alpha=0.7, codes=codes), 20)
            byt = (1 << 28) * (4 + 4 / (32 // b))
            out.append({"project": 1 << 28, "fmt": [b, k], "us": round(us, 1), "GB/s": round(byt / us / 1e3, 1),
                        "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
    del x
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
    codes + output codes (+ weights, scale and bias).  Each call reads the next
    of several input copies (over 3 x L2 in total), so inputs come from HBM;
    codes are uniformly drawn words (timing only)."""
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(0)
    fx, fw = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)
    n = 64
    span = 3 * 129 * 10 ** 6

    def copies(rows, ld, unsigned):
        nbytes = rows * ld * 4
        nx = max(1, min(256, -(-span // nbytes)))
        c = torch.randint(0, 2 ** 32, (nx * rows, ld), generator=g, device=dev, dtype=torch.int64).to(torch.int32)
        if unsigned:
            c &= 0x77777777
        return [c[i * rows:(i + 1) * rows] for i in range(nx)], nbytes

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
        it = [0]

        def f():
            X = Xs[it[0] % len(Xs)]
            it[0] += 1
            esb.esb_conv2d_nhwc(X, fx, W, fw, n, h, h, c, c, 3, 3, stride, 1, groups=c, ep=ep, want_acc=False,
                                want_codes=True, out_codes=oc)

        us = timeit(f, 20)
        byt = xb + oc.numel() * 4 + W.numel() * 4 + 8 * c
        res.append({"dwconv": [n, h, h, c, stride], "fmt": [4, 2], "us": round(us, 2),
                    "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
        del Xs, oc
    Xs, xb = copies(n * 112 * 112, 8, True)
    Y = torch.empty((n * 56 * 56, 8), dtype=torch.int32, device=dev)
    it = [0]

    def mp():
        esb.esb_maxpool_nhwc(Xs[it[0] % len(Xs)], fx, n, 112, 112, 64, 3, 2, 1, out=Y)
        it[0] += 1

    us = timeit(mp, 20)
    byt = xb + Y.numel() * 4
    res.append({"maxpool": [n, 112, 112, 64, 3, 2], "fmt": [4, 2], "us": round(us, 2),
                "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
    del Xs, Y
    for c in (512, 1280):
        ld = esb.esb_row_words(c, 4)
        Xs, xb = copies(n * 49, ld, True)
        it = [0]

        def ap():
            esb.esb_avgpool_nhwc(Xs[it[0] % len(Xs)], fx, n, 49, c, 1.0 / 49, 0.5, fx)
            it[0] += 1

        us = timeit(ap, 20)
        byt = xb + n * ld * 4
        res.append({"avgpool": [n, 7, 7, c], "fmt": [4, 2], "us": round(us, 2),
                    "GB/s": round(byt / us / 1e3, 1), "frac_hbm": round(byt / us / 1e3 / hbm, 3)})
        del Xs
    res.append({"cc_status": esb.esb_get_status()})
    return res


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweeps", nargs="?", const="all", choices=["all", "gemm", "project", "cc"],
                    help="the sweeps instead of the step (all, or only the GEMM, projection or CUDA-core part)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.sweeps:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()

#!/usr/bin/env python
"""Benchmark of the sparsity/intensity-dispatched operator path on GB300.

Default workload (one step = one pass of the per-operator hot path over one
batch): the 3x3 convolution NHWC bf16 [8, 56, 56, 64] -> 64 channels, stride 1,
pad 1, input ReLU(N(0,1)) (about half zeros), BN + ReLU epilogue:
  1. Eq. 1 statistics and occupancy bitmaps of the input (stats kernel),
  2. Eq. 2 work as FLOPs per input byte (host arithmetic on the shape),
  3. threshold dispatch on the device (s_thr 0.5, c_thr 32 FLOP/B),
  4. the chosen tcgen05 kernel (dense or zero-skip) with the fused epilogue,
     which also writes the output's occupancy for the next operator.
Metric: effective TFLOP/s = dense-equivalent FLOPs / time.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl sparoa|reference]
       [--workload conv|fc|resnet18|mobilenet_v2|vit_b16|mlp_sweep|ops|calibrate|batching|split]
       [--batch B]
       [--thresholds default|calibrated] [--calib-out PATH]
For N > 1 launch one process per GPU with torch.distributed.run; every rank
runs its own replica (weak scaling), timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "effective TFLOP/s & % roofline per op; synthetic CNN images/s at batch 1/32"
NBUF = 40   # rotating input/output sets per step, 40 x 6.6 MB > 129 MB L2
# one sparoa_conv2d call measuring its own input: a small clear (the input's
# counters and block masks), the stats kernel (which also zeroes the output's
# occupancy block) and the conv kernel
LAUNCHES_PER_CONV_STEP = 3


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=60000)
    p.add_argument("--warmup", type=int, default=400)
    p.add_argument("--impl", default="sparoa", choices=["sparoa", "reference"])
    p.add_argument("--workload", default="conv",
                   choices=["conv", "fc", "resnet18", "mobilenet_v2", "vit_b16", "mlp_sweep", "ops",
                            "calibrate", "batching", "split", "profile"])
    p.add_argument("--op", default="conv_cfg2",
                   help="profile: the operator to run (see run_profile)")
    p.add_argument("--batch", type=int, default=32)
    p.add_argument("--thresholds", default="default", choices=["default", "calibrated"],
                   help="graph workloads: the default s_thr/c_thr, or the per-operator thresholds "
                        "of the committed calibration table")
    p.add_argument("--calib-out", default=None, help="calibrate: write the thresholds table here")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-extras", action="store_true",
                   help="conv workload: skip the other configurations' sub-records")
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "sm_max_mhz": d.get("sm_max_mhz"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sm_max_mhz": 2070.0, "source": "fallback"}


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.samples = []
        self.proc = None
        self.marks = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [s.strip() for s in line.split(",")]
            if len(parts) >= 8:
                self.samples.append((time.time(), parts))

    def mark(self):
        self.marks.append(time.time())

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        def num(s):
            try:
                return float(s)
            except ValueError:
                return None
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}
        t0, t1 = (self.marks[0], self.marks[-1]) if len(self.marks) >= 2 else (0, 1e30)
        inside = [p for t, p in self.samples if t0 <= t <= t1] or [p for _, p in self.samples]
        sm = [num(p[0]) for p in inside if num(p[0]) is not None]
        mx = [num(p[1]) for p in inside if num(p[1]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for p in inside for n, v in zip(names, p[4:8]) if v.lower() == "active"})
        pw = [num(p[2]) for p in inside if num(p[2]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "power_w_max": max(pw) if pw else None, "samples": len(inside)}


# ---------------------------------------------------------------------------
# distributed helpers (one process per GPU; no data-path collective)
# ---------------------------------------------------------------------------
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), \
        int(os.environ.get("WORLD_SIZE", 1))


def max_over_ranks(value: float, world: int, device):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# The sources a captured kernel is compiled from: its own file and the shared
# device headers.  A capture stays valid while these are unchanged.
KERNEL_SOURCES = {
    "conv3_kernel_8x56x56x64": ["k_conv3.cu"],
    "stats_kernel_25088x64": ["k_tiles.cu"],
    "igemm_kernel_4096x3072x768": ["k_igemm.cu"],
}
COMMON_SOURCES = ["sparoa_dev.cuh", "sparoa_kernels.h"]


def kernel_source_hash(key: str) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2511_19457_gb300", "csrc")
    for f in COMMON_SOURCES + KERNEL_SOURCES[key]:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(key: str):
    """Per-launch DRAM bytes of `key` from the committed ncu summary, or None
    when the kernels changed since that capture."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    e = d.get(key)
    if not e or key not in KERNEL_SOURCES or e.get("kernel_source_sha") != kernel_source_hash(key):
        return None
    return e.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------
# CPU baseline: the oracle as it stands, on the host cores
# ---------------------------------------------------------------------------
def oracle_conv_step(d):
    from oracle import oracle as orc
    N, H, W, C = d["N"], d["H"], d["W"], d["Cin"]
    st = orc.stats(d["x"], N * H * W, C)
    wk = orc.conv_work(N, H, W, C, d["Cout"], 3, 3, 1, 1)
    path = orc.decide(st.numel, st.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0)
    y = orc.conv2d(d["x"], N, H, W, C, d["w"], d["Cout"], 3, 3, 1, 1, bn=d["bn"], act=1,
                   skip_zeros=(path == 2))
    bits = orc.f64_to_bf16(y)
    orc.stats(bits, N * H * W, d["Cout"])
    return wk.flops


def cpu_baseline_conv(budget_s: float = 10.0, min_reps: int = 2):
    from oracle import oracle as orc
    from paper_2511_19457_gb300 import synth
    d = synth.conv_layer(seed=0)
    oracle_conv_step(d)  # load / first touch
    reps, flops, t0 = 0, 0, time.perf_counter()
    while reps < min_reps or time.perf_counter() - t0 < budget_s:
        flops += oracle_conv_step(d)
        reps += 1
    dt = time.perf_counter() - t0
    return {"value": flops / dt / 1e12, "unit": "TFLOP/s", "cores": orc.num_threads(),
            "kind": "oracle",
            "sample": f"{reps} full passes of the conv workload (stats, rule, fp64 direct conv, "
                      f"bf16 rounding, output stats) in {dt:.1f} s"}


# ---------------------------------------------------------------------------
# the reference arm: the oracle, timed on the host
# ---------------------------------------------------------------------------
def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return 0
    from oracle import oracle as orc
    from paper_2511_19457_gb300 import synth
    d = synth.conv_layer(seed=0)
    for _ in range(max(args.warmup, 0)):
        oracle_conv_step(d)
    steps = max(args.steps, 1)
    t0 = time.perf_counter()
    flops = 0
    for _ in range(steps):
        flops += oracle_conv_step(d)
    dt = time.perf_counter() - t0
    v = flops / dt / 1e12
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": args.gpus,
            "steps": steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": conv_config(),
            "cpu_baseline": {"kind": "oracle", "cores": orc.num_threads(),
                             "sample": f"{steps} full passes of the conv workload per timed region",
                             "value": v, "unit": "TFLOP/s"},
            "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def conv_config():
    return {"workload": "conv3x3 s1 p1 NHWC bf16 [8,56,56,64]->64, BN+ReLU epilogue; "
                        "Eq.1 stats + threshold dispatch + next-op occupancy",
            "global_batch": 8, "seq_len": None, "parallelism": "replicas",
            "thresholds": {"s_thr": 0.5, "c_thr_flops_per_byte": 32.0},
            "l2": f"GPU arm: {NBUF} rotating input/output sets (257 MB > 129 MB L2)"}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def graph_of(fn, count):
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for j in range(count):
            fn(j)
    return g


def time_graph(g, replays):
    import torch
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(replays):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1)


def time_graph_per_replay(g, min_replays=50, min_s=0.2, max_replays=20000):
    """ms per replay over at least `min_replays` replays and `min_s` seconds
    (a short probe sizes the run); independent of the bench's --steps."""
    probe = time_graph(g, 5) / 5
    reps = max(min_replays, int(math.ceil(min_s * 1e3 / max(probe, 1e-6))))
    reps = min(reps, max_replays)
    return time_graph(g, reps) / reps, reps


def run_conv(args, rank, local_rank, world, peaks):
    import numpy as np
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    d = synth.conv_layer(seed=0)
    N, H, W, C, Co = 8, 56, 56, 64, 64
    R = N * H * W
    x0 = sp.bits_to_device(d["x"]).view(N, H, W, C)
    xs = [x0.clone() for _ in range(NBUF)]
    w = sp.bits_to_device(d["w"]).view(Co, 3, 3, C)
    bn = torch.from_numpy(d["bn"]).to(dev)
    ys = [torch.empty(N, H, W, Co, dtype=torch.bfloat16, device=dev) for _ in range(NBUF)]
    xo = [sp.OccupancyBuffer(R, C) for _ in range(NBUF)]
    yo = [sp.OccupancyBuffer(R, Co) for _ in range(NBUF)]
    thr = sp.thresholds()
    flops = 2 * N * H * W * Co * C * 9

    def stats(j):
        sp.sparoa_op_stats(ctx, xs[j], (N, H, W, C), occ=xo[j], host=False)

    def conv(j):
        sp.sparoa_conv2d(ctx, xs[j], w, ys[j], stride=1, pad=1, bn=bn, act=sp.ACT_RELU, thr=thr,
                         x_occ=xo[j], y_occ=yo[j])

    def step(j):
        # one call: the input's Eq. 1 statistics measured inside it (a small
        # clear, the stats kernel), then the dispatched conv kernel
        sp.sparoa_conv2d(ctx, xs[j], w, ys[j], stride=1, pad=1, bn=bn, act=sp.ACT_RELU, thr=thr,
                         y_occ=yo[j])

    # path actually taken and the occupied share of K blocks (algorithmic work)
    st = sp.sparoa_conv2d(ctx, xs[0], w, ys[0], stride=1, pad=1, bn=bn, act=sp.ACT_RELU, thr=thr,
                          host=True)
    path = "zero-skip" if st.path == sp.PATH_SKIP else "dense"
    occ_frac = 1.0
    if st.path == sp.PATH_SKIP:
        sp.sparoa_op_stats(ctx, xs[0], (N, H, W, C), occ=xo[0], host=False)
        occ_frac = conv_occupied_fraction(xo[0].to_host(), N, H, W, C)

    for j in range(max(args.warmup, 3)):
        step(j % NBUF)
    torch.cuda.synchronize()
    g_full = graph_of(step, NBUF)
    rem = args.steps % NBUF
    g_rem = graph_of(step, rem) if rem else None
    g_full.replay()
    torch.cuda.synchronize()

    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    clocks = ClockSampler(int(vis.split(",")[local_rank]) if vis else local_rank)
    clocks.start()
    time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize()
    clocks.mark()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps // NBUF):
        g_full.replay()
    if g_rem is not None:
        g_rem.replay()
    e1.record()
    torch.cuda.synchronize()
    clocks.mark()
    ms = e0.elapsed_time(e1)
    barrier(world)
    ms = max_over_ranks(ms, world, dev)

    # per-kernel durations (same launches, same buffers), measured live over
    # >= 50 replays and >= 0.2 s whatever --steps is
    g_stats = graph_of(stats, NBUF)
    g_conv = graph_of(conv, NBUF)
    g_stats.replay()
    g_conv.replay()
    clocks.mark()
    ms_r, stats_reps = time_graph_per_replay(g_stats)
    stats_us = ms_r * 1e3 / NBUF
    ms_r, conv_reps = time_graph_per_replay(g_conv)
    conv_us = ms_r * 1e3 / NBUF
    clocks.mark()
    clocks.stop()

    # end to end through the public API: every step copies its input from pinned
    # host memory, runs, and copies its output back to pinned host memory.  The
    # copies run on their own streams, so step j's input copy and step j-1's
    # output copy overlap step j's compute, as in a serving pipeline; all of
    # them are inside the timed graph.
    xh = torch.from_numpy(d["x"].view(np.int16)).view(torch.bfloat16).view(N, H, W, C).pin_memory()
    yhs = [torch.empty(N, H, W, Co, dtype=torch.bfloat16).pin_memory() for _ in range(NBUF)]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()

    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e):
        cap = torch.cuda.current_stream()
        s_in.wait_stream(cap)
        s_out.wait_stream(cap)
        for j in range(NBUF):
            ev_in, ev_done = torch.cuda.Event(), torch.cuda.Event()
            with torch.cuda.stream(s_in):
                xs[j].copy_(xh, non_blocking=True)
                ev_in.record(s_in)
            cap.wait_event(ev_in)
            step(j)
            ev_done.record(cap)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_done)
                yhs[j].copy_(ys[j], non_blocking=True)
        cap.wait_stream(s_in)
        cap.wait_stream(s_out)
    g_e2e.replay()
    e2e_reps = max(1, min(args.steps // NBUF, 250))
    e2e_ms = time_graph(g_e2e, e2e_reps)
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    e2e_steps = e2e_reps * NBUF

    # the roofline of the dominant kernel (the conv; stats kernel also reported)
    alg_flops = flops * occ_frac
    conv_bytes = (R * C + R * Co + Co * 9 * C) * 2 + 2 * int(sp._lib.sparoa_occupancy_bytes(R, Co))
    achieved_tf = alg_flops / (conv_us * 1e-6) / 1e12
    stats_bytes = R * C * 2 + int(sp._lib.sparoa_occupancy_bytes(R, C))
    roof = {"bound": "tensor", "achieved": achieved_tf, "peak": peaks["bf16_tflops"],
            "unit": "TFLOP/s", "frac": achieved_tf / peaks["bf16_tflops"],
            "traffic": ncu_traffic("conv3_kernel_8x56x56x64"),
            "kernel": "conv3_kernel<64> (" + path + ")", "kernel_us": conv_us,
            "algorithmic_flops": alg_flops, "algorithmic_bytes": conv_bytes,
            "hbm_view": {"achieved_gbs": conv_bytes / (conv_us * 1e-6) / 1e9,
                         "frac": conv_bytes / (conv_us * 1e-6) / 1e9 / peaks["hbm_gbs"]},
            "peak_source": peaks["source"]}
    stats_kernel = {"kernel": "stats_kernel", "kernel_us": stats_us, "bytes": stats_bytes,
                    "achieved_gbs": stats_bytes / (stats_us * 1e-6) / 1e9,
                    "frac_hbm": stats_bytes / (stats_us * 1e-6) / 1e9 / peaks["hbm_gbs"]}

    total_flops = flops * args.steps * world
    value = total_flops / (ms * 1e-3) / 1e12
    e2e_value = flops * e2e_steps * world / (e2e_ms * 1e-3) / 1e12
    cfg = conv_config()
    detail = {"path": path, "rho": st.sparsity, "occupied_k_fraction": occ_frac,
              "rotating_sets_mb": round(NBUF * 2 * R * C * 2 / 1e6), "cuda_graph": True,
              "replicas": world, "kernel_timing_replays": {"stats": stats_reps * NBUF,
                                                           "conv": conv_reps * NBUF}}
    line = {"metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded; stands in for ImageNet activations)", "config": cfg,
            "workload_detail": detail, "roofline": roof, "stats_kernel": stats_kernel,
            "e2e": {"value": e2e_value, "unit": "TFLOP/s", "h2d_bytes_per_step": R * C * 2,
                    "d2h_bytes_per_step": R * Co * 2, "steps": e2e_steps,
                    "copies": "pinned host <-> device on two side streams, overlapping compute"},
            # per step: one clear (input and output occupancy), stats kernel, conv kernel
            "gpu_launches": LAUNCHES_PER_CONV_STEP * args.steps,
            "clocks": clocks.summary()}
    ctx.close()
    return line


def conv_occupied_fraction(occ, N, H, W, C, k=3, pad=1):
    """Share of (128-pixel M tile, tap, 32-channel block) K slices the zero-skip
    kernel must stage: a slice is left out when none of the tile's 128 shifted
    input pixels has an occupied 64-channel tile there."""
    import numpy as np
    T = (C + 63) // 64
    bm = occ["row_bm"].reshape(N, H, W, -1)
    tile_occ = np.stack([((bm[..., t // 64] >> np.uint64(t % 64)) & np.uint64(1)).astype(bool)
                         for t in range(T)], axis=-1)            # [N, H, W, T]
    M = N * H * W
    m = np.arange(M)
    n, oh, ow = m // (H * W), (m // W) % H, m % W
    cb = (C + 31) // 32
    total = occupied = 0
    for r in range(k):
        for s in range(k):
            ih, iw = oh - pad + r, ow - pad + s
            ok = (ih >= 0) & (ih < H) & (iw >= 0) & (iw < W)
            vals = np.zeros((M, T), dtype=bool)
            vals[ok] = tile_occ[n[ok], ih[ok], iw[ok]]
            tiles = vals.reshape(-1, 128, T) if M % 128 == 0 else None
            if tiles is None:
                pad_rows = (-M) % 128
                tiles = np.concatenate([vals, np.zeros((pad_rows, T), bool)]).reshape(-1, 128, T)
            any_t = tiles.any(axis=1)                              # [tiles, T]
            for b in range(cb):
                total += any_t.shape[0]
                occupied += int(any_t[:, (b * 32) // 64].sum())
    return occupied / total if total else 1.0


def fc_record(ctx, dev, peaks):
    """The single FC operator [64, 512] x [512, 512]^T (column-sparse ReLU
    input, fp32 output): one step = one sparoa_gemm call (the input's Eq. 1
    count measured inside it, dispatch, the chosen kernel) over rotating
    input / output sets; roofline HBM-bound: occupied weight rows + x + y."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    d = synth.fc_layer(seed=0)
    M, K, N = d["M"], d["K"], d["N"]
    xs = [sp.bits_to_device(d["x"]).view(M, K).clone() for _ in range(NBUF)]
    w = sp.bits_to_device(d["w"]).view(N, K)
    wkn = sp.bits_to_device(d["w_kn"]).view(K, N)
    bias = torch.from_numpy(d["bias"]).to(dev)
    ys = [torch.empty(M, N, dtype=torch.float32, device=dev) for _ in range(NBUF)]
    def step(j):
        # one call: the input's Eq. 1 count measured inside it, dispatch, FC
        sp.sparoa_gemm(ctx, xs[j], w, ys[j], W_kn=wkn, bias=bias)

    st = sp.sparoa_gemm(ctx, xs[0], w, ys[0], W_kn=wkn, bias=bias, host=True)
    for j in range(NBUF):
        step(j)
    g_step = graph_of(step, NBUF)
    g_step.replay()
    step_ms, _ = time_graph_per_replay(g_step)
    step_us = gemm_us = step_ms * 1e3 / NBUF
    kocc = int((xs[0].float().abs().sum(0) != 0).sum().item())
    flops = 2 * M * K * N
    alg_bytes = (kocc * N * 2 + M * K * 2 + M * N * 4) if st.path == sp.PATH_SKIP else (N * K + M * K) * 2 + M * N * 4
    ach = alg_bytes / (gemm_us * 1e-6) / 1e9
    return {"workload": "fc [64,512]x[512,512]^T fp32 out, ReLU input with whole columns zeroed "
                        "(p=0.4), s_thr 0.5",
            "path": PATH_NAME.get(int(st.path)), "rho": st.sparsity, "occupied_k": kocc,
            "step_us": step_us, "step_tflops": flops / (step_us * 1e-6) / 1e12,
            "roofline": {"bound": "hbm", "kernel": "sparoa_gemm call: fused small-FC kernel (count, "
                                                   "dispatch, zero-skip product) + the dense kernel's exit",
                         "kernel_us": gemm_us, "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": ach / peaks["hbm_gbs"], "algorithmic_bytes": alg_bytes,
                         "note": "weights shared by the rotating sets (L2-resident across calls)"}}


def graphs_record(ctx, steps=30):
    """ResNet-18 at batch 1 / 8 / 32 and MobileNetV2 at batch 1 / 32 through
    sparoa_run_graph (CUDA graph, L2 flushed before every timed replay)."""
    out = {}
    for name, batch in [("resnet18", 1), ("resnet18", 8), ("resnet18", 32),
                        ("mobilenet_v2", 1), ("mobilenet_v2", 32)]:
        ms, recs = time_graph_workload(ctx, name, batch, steps, 3)
        flops = sum(r.stats.flops for r in recs)
        paths = [int(r.stats.path) for r in recs]
        out[f"{name}_b{batch}"] = {
            "images_per_s": batch / (ms * 1e-3), "ms_per_batch": ms,
            "effective_tflops": flops / (ms * 1e-3) / 1e12,
            "ops": {"dense": paths.count(1), "zero_skip": paths.count(2), "depthwise": paths.count(3),
                    "other": paths.count(0)},
            "decisions": [(int(r.stats.numel), int(r.stats.nnz), float(r.stats.flops_per_byte),
                           int(r.stats.macs_eq2), int(r.stats.path)) for r in recs]}
    return out


def ops_cfg4_record(ctx, dev, peaks):
    """Dense tcgen05 path at MobileNetV2's (batch 32) stem, expansion,
    projection, last pointwise and classifier shapes: the conv / FC call with
    the dense path forced, input occupancy measured beforehand, rotating
    input / output sets larger than L2."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    gen = torch.Generator(device=dev).manual_seed(1)
    tc = peaks["bf16_tflops"]
    rows = []
    shapes = [("stem 3x3 s2", 32, 224, 224, 3, 32, 3, 2, 1),
              ("expand 1x1", 32, 56, 56, 24, 144, 1, 1, 0),
              ("project 1x1", 32, 56, 56, 144, 24, 1, 1, 0),
              ("expand 1x1", 32, 28, 28, 32, 192, 1, 1, 0),
              ("project 1x1", 32, 14, 14, 384, 64, 1, 1, 0),
              ("expand 1x1", 32, 14, 14, 64, 384, 1, 1, 0),
              ("last 1x1", 32, 7, 7, 320, 1280, 1, 1, 0)]
    for tag, N, H, W, C, Co, k, s_, p_ in shapes:
        Ho, Wo = (H + 2 * p_ - k) // s_ + 1, (W + 2 * p_ - k) // s_ + 1
        in_b = N * H * W * C * 2
        nb = max(2, min(40, int(3 * 129e6 / (in_b + N * Ho * Wo * Co * 2)) + 1))
        w = (torch.randn(Co, k, k, C, device=dev, generator=gen) / math.sqrt(k * k * C)).to(torch.bfloat16)
        xs = []
        for _ in range(nb):
            v = torch.randn(N, H, W, C, device=dev, generator=gen).clamp_min_(0.0)
            xs.append(v.to(torch.bfloat16))
        ys = [torch.empty(N, Ho, Wo, Co, dtype=torch.bfloat16, device=dev) for _ in range(nb)]
        xo = [sp.OccupancyBuffer(N * H * W, C) for _ in range(nb)]
        for j in range(nb):
            sp.sparoa_op_stats(ctx, xs[j], (N, H, W, C), occ=xo[j], host=False)
        dense = sp.thresholds(force_path=sp.PATH_DENSE)
        call = lambda j: sp.sparoa_conv2d(ctx, xs[j], w, ys[j], stride=s_, pad=p_, act=sp.ACT_RELU6,
                                          thr=dense, x_occ=xo[j])
        for j in range(nb):
            call(j)
        g = graph_of(call, nb)
        g.replay()
        ms, _ = time_graph_per_replay(g)
        us = ms * 1e3 / nb
        flops = 2.0 * N * Ho * Wo * Co * C * k * k
        rule = sp.sparoa_conv2d(ctx, xs[0], w, ys[0], stride=s_, pad=p_, act=sp.ACT_RELU6, host=True)
        ach = flops / (us * 1e-6) / 1e12
        rows.append({"op": f"{tag} [{N},{H},{W},{C}]->{Co}", "us": round(us, 2), "bound": "tensor",
                     "achieved": round(ach, 1), "unit": "TFLOP/s", "peak": tc, "frac": round(ach / tc, 4),
                     "flop_per_byte": round(float(rule.flops_per_byte), 1),
                     "rule_path": PATH_NAME.get(int(rule.path)), "rotating_sets": nb})
        del xs, ys, xo, g
        torch.cuda.empty_cache()
    return rows


def mlp_sweep_record(ctx, dev, rhos=None, structures=("unstructured", "block32", "token")):
    """The MLP down projection h [M, 3072] x W2 [768, 3072]^T at M in {256,
    1024, 4096}: forced-dense and forced-zero-skip time per zero fraction rho
    and zero structure, the crossover rho (the smallest rho from which
    zero-skip is faster at every larger rho of the grid), and what the rule
    (s_thr 0.5, c_thr 32) picks on the measured count.  Each point's input is
    drawn once (seeded) and copied into rotating sets larger than L2."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    wts = synth.mlp_weights(seed=0)
    w2 = sp.bits_to_device(wts["w2"]).view(768, 3072)
    rhos = rhos or [round(0.05 * i, 2) for i in range(20)]
    table, cross = [], {}
    for M in (256, 1024, 4096):
        nb = max(2, int(3 * 129e6 / (M * 3072 * 2 + M * 768 * 2)) + 1)
        ys = [torch.empty(M, 768, dtype=torch.bfloat16, device=dev) for _ in range(nb)]
        for structure in structures:
            wins = []
            for rho in rhos:
                h0 = sp.bits_to_device(synth.mlp_hidden(M, rho, structure, seed=M)).view(M, 3072)
                hs = [h0] + [h0.clone() for _ in range(nb - 1)]
                occ = [sp.OccupancyBuffer(M, 3072) for _ in range(nb)]
                for j in range(nb):
                    sp.sparoa_op_stats(ctx, hs[j], (M, 3072), occ=occ[j], host=False)
                times = {}
                for force in (1, 2):
                    thr = sp.thresholds(force_path=force)
                    g = graph_of(lambda j: sp.sparoa_gemm(ctx, hs[j], w2, ys[j], thr=thr, x_occ=occ[j]), nb)
                    g.replay()
                    ms, _ = time_graph_per_replay(g, min_replays=10, min_s=0.02)
                    times[force] = ms * 1e3 / nb
                rule = sp.sparoa_gemm(ctx, hs[0], w2, ys[0], x_occ=occ[0], host=True)
                table.append({"M": M, "structure": structure, "rho": rho, "nnz": int(rule.nnz),
                              "dense_us": round(times[1], 2), "skip_us": round(times[2], 2),
                              "rule_path": PATH_NAME.get(int(rule.path))})
                wins.append(times[2] < times[1])
                del hs, occ
            crossover = None
            for i in range(len(rhos) - 1, -1, -1):
                if not wins[i]:
                    break
                crossover = rhos[i]
            cross[f"M{M}_{structure}"] = crossover
        del ys
        torch.cuda.empty_cache()
    return {"workload": "MLP down projection [M,3072]x[768,3072]^T, bf16, M in {256,1024,4096}",
            "crossover_rho": cross, "rule": {"s_thr": 0.5, "c_thr": 32.0, "flop_per_byte": 768.0},
            "table": table}


def other_configs(ctx, dev, peaks):
    """The other configurations of the metric, as sub-records of the default
    line: the FC operator, the two CNNs at batch 1 / 8 / 32, MobileNetV2's
    dense-path shapes and the MLP sparsity sweep."""
    out = {}
    for key, fn in [("fc", lambda: fc_record(ctx, dev, peaks)),
                    ("graphs", lambda: graphs_record(ctx)),
                    ("mobilenet_v2_dense_ops", lambda: ops_cfg4_record(ctx, dev, peaks)),
                    ("mlp_sweep", lambda: mlp_sweep_record(ctx, dev))]:
        t0 = time.perf_counter()
        try:
            out[key] = fn()
        except Exception as e:  # a failed sub-record must not lose the headline line
            out[key] = {"error": f"{type(e).__name__}: {e}"}
        out.setdefault("seconds", {})[key] = round(time.perf_counter() - t0, 1)
    return out


def oracle_rule_check(extra):
    """The oracle's threshold rule on the counts the device measured (the
    CPU-baseline leg): agreement of every recorded dispatch decision."""
    from oracle import oracle as orc
    n = agree = 0
    sweep = extra.get("mlp_sweep", {})
    for row in sweep.get("table", []):
        want = orc.decide(row["M"] * 3072, row["nnz"], 768.0, 3072 * 768, 0.5, 32.0)
        n += 1
        agree += int(PATH_NAME.get(want) == row["rule_path"])
    for rec in extra.get("graphs", {}).values():
        if not isinstance(rec, dict):
            continue
        for numel, nnz, fpb, macs, path in rec.get("decisions", []):
            if path in (1, 2):
                n += 1
                agree += int(orc.decide(numel, nnz, fpb, macs, 0.5, 32.0) == path)
    return {"decisions_checked": n, "agree": agree}


def run_fc(args, rank, local_rank, world, peaks):
    """Single FC operator [64, 512] x [512, 512]^T (column-sparse ReLU input),
    fp32 output: stats + dispatch + the chosen kernel, CUDA-graph replays."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    d = synth.fc_layer(seed=0)
    M, K, N = d["M"], d["K"], d["N"]
    nb = NBUF
    xs = [sp.bits_to_device(d["x"]).view(M, K).clone() for _ in range(nb)]
    w = sp.bits_to_device(d["w"]).view(N, K)
    wkn = sp.bits_to_device(d["w_kn"]).view(K, N)
    bias = torch.from_numpy(d["bias"]).to(dev)
    ys = [torch.empty(M, N, dtype=torch.float32, device=dev) for _ in range(nb)]
    xo = [sp.OccupancyBuffer(M, K) for _ in range(nb)]

    def step(j):
        sp.sparoa_op_stats(ctx, xs[j], (M, K), occ=xo[j], host=False)
        sp.sparoa_gemm(ctx, xs[j], w, ys[j], W_kn=wkn, bias=bias, x_occ=xo[j])

    st = sp.sparoa_gemm(ctx, xs[0], w, ys[0], W_kn=wkn, bias=bias, host=True)
    for j in range(max(args.warmup, 3)):
        step(j % nb)
    g = graph_of(step, nb)
    g.replay()
    reps = max(1, args.steps // nb)
    ms = time_graph(g, reps) / (reps * nb)
    ms = max_over_ranks(ms, world, dev)
    flops = 2 * M * K * N
    ctx.close()
    return {"metric": METRIC, "value": flops * world / (ms * 1e-3) / 1e12, "unit": "TFLOP/s",
            "n_gpus": world, "steps": reps * nb, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "config": {"workload": "fc [64,512]x[512,512] fp32 out, column-sparse "
                                            "ReLU input (rho ~0.7), stats + dispatch",
                                            "path": "zero-skip" if st.path == sp.PATH_SKIP else "dense",
                                            "rho": st.sparsity}}


def run_mlp_sweep(args, rank, local_rank, world, peaks):
    """Down projection of a 768 -> 3072 -> 768 ReLU MLP, h [M, 3072] x W2 [768, 3072]^T,
    at activation sparsity 0..0.95: dense tcgen05 vs zero-skip time per point, the
    crossover sparsity where zero-skip wins, and what the rule (s_thr 0.5) picks."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    wts = synth.mlp_weights(seed=0)
    w2 = sp.bits_to_device(wts["w2"]).view(768, 3072)
    rhos = [round(0.05 * i, 2) for i in range(20)]
    table = []
    cross = {}
    for M in (256, 1024, 4096):
        for structure in ("unstructured", "block32"):
            nb = 4 if M == 4096 else 8
            y = torch.empty(M, 768, dtype=torch.bfloat16, device=dev)
            crossover = None
            for rho in rhos:
                hs = [sp.bits_to_device(synth.mlp_hidden(M, rho, structure, seed=j)).view(M, 3072)
                      for j in range(nb)]
                occ = [sp.OccupancyBuffer(M, 3072) for _ in range(nb)]
                for j in range(nb):
                    sp.sparoa_op_stats(ctx, hs[j], (M, 3072), occ=occ[j], host=False)
                times = {}
                for force in (1, 2):
                    thr = sp.thresholds(force_path=force)
                    g = graph_of(lambda j: sp.sparoa_gemm(ctx, hs[j], w2, y, thr=thr, x_occ=occ[j]), nb)
                    g.replay()
                    times[force] = time_graph(g, 10) / (10 * nb)
                rule = sp.sparoa_gemm(ctx, hs[0], w2, y, x_occ=occ[0], host=True)
                fl = 2 * M * 3072 * 768
                row = {"M": M, "structure": structure, "rho": rho, "measured_rho": rule.sparsity,
                       "dense_us": times[1] * 1e3, "skip_us": times[2] * 1e3,
                       "dense_tflops": fl / (times[1] * 1e-3) / 1e12,
                       "skip_eff_tflops": fl / (times[2] * 1e-3) / 1e12,
                       "rule_path": "zero-skip" if rule.path == sp.PATH_SKIP else "dense"}
                table.append(row)
                if crossover is None and times[2] < times[1]:
                    crossover = rho
                del hs, occ
            cross[f"M{M}_{structure}"] = crossover
    ctx.close()
    return {"metric": METRIC, "value": None, "unit": "us per down-projection", "n_gpus": world,
            "higher_is_better": False, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "MLP down projection [M,3072]x[768,3072]^T sparsity sweep"},
            "crossover_rho": cross, "table": table}


def time_graph_workload(ctx, name, batch, steps, warmup, thresholds="default"):
    """ms per replay of one CUDA-graph-captured sparoa_run_graph over the
    synthetic CNN, the L2 flushed before every replay; returns (ms, records)."""
    import torch

    from paper_2511_19457_gb300 import calibrate as cal
    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", ctx.device)
    ops, xb, shape = {"resnet18": synth.resnet18, "mobilenet_v2": synth.mobilenet_v2,
                      "vit_b16": synth.vit}[name](batch=batch)
    if thresholds == "calibrated":
        ops = cal.apply(ops, shape, cal.load_table())
    elif isinstance(thresholds, dict):
        ops = cal.apply(ops, shape, thresholds)
    graph = sp.Graph(ops)
    x = sp.bits_to_device(xb).view(*shape)
    recs = sp.sparoa_run_graph(ctx, graph, x, records=True)
    for _ in range(max(warmup, 3)):
        sp.sparoa_run_graph(ctx, graph, x)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        sp.sparoa_run_graph(ctx, graph, x)
    g.replay()
    # a small batch fits in L2: before every replay a 256 MB write evicts it,
    # outside the events that time the replay
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(steps)]
    torch.cuda.synchronize()
    for e0, e1 in evs:
        flush.zero_()
        e0.record()
        g.replay()
        e1.record()
    torch.cuda.synchronize()
    ms = sum(e0.elapsed_time(e1) for e0, e1 in evs) / steps
    del g, flush
    return ms, recs


PATH_NAME = {0: "none", 1: "dense", 2: "zero-skip", 3: "depthwise"}


def run_graph_workload(args, rank, local_rank, world, peaks, name):
    """CNN images/s through sparoa_run_graph (not the default bench line)."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    ms, recs = time_graph_workload(ctx, name, args.batch, args.steps, args.warmup, args.thresholds)
    flops = sum(r.stats.flops for r in recs)
    ms = max_over_ranks(ms, world, dev)
    ops_table = [{"op": i, "path": PATH_NAME.get(int(r.stats.path), str(int(r.stats.path))),
                  "rho": round(float(r.stats.sparsity), 4), "gflop": round(r.stats.flops / 1e9, 4),
                  "flop_per_byte": round(float(r.stats.flops_per_byte), 1)}
                 for i, r in enumerate(recs)]
    line = {"metric": METRIC, "value": args.batch * world / (ms * 1e-3), "unit": "images/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "effective_tflops": flops / (ms * 1e-3) / 1e12,
            "config": {"workload": f"{name} B={args.batch} through sparoa_run_graph (CUDA graph)",
                       "thresholds": args.thresholds,
                       "global_batch": args.batch * world,
                       "l2": "flushed by a 256 MB write before every timed replay"},
            "ops": ops_table}
    ctx.close()
    return line


def run_ops(args, rank, local_rank, world, peaks):
    """Per-operator roofline: every kernel of the path at the workloads' shapes,
    timed as CUDA-graph replays over rotating input/output sets larger than L2;
    achieved = algorithmic bytes (or dense-equivalent FLOPs) / time per call."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    gen = torch.Generator(device=dev).manual_seed(0)
    L2 = 129e6
    hbm, tc = peaks["hbm_gbs"], peaks["bf16_tflops"]
    occ_b = lambda R, C: int(sp._lib.sparoa_occupancy_bytes(R, C))

    def act_like(*shape, zero_p=0.5):
        v = torch.randn(*shape, device=dev, generator=gen).abs()
        v[torch.rand(*shape, device=dev, generator=gen) < zero_p] = 0.0
        return v.to(torch.bfloat16)

    rows = []

    def measure(name, make_set, call, set_bytes, alg_bytes=0.0, alg_flops=0.0, bound="hbm"):
        nb = max(2, min(40, int(3 * L2 / max(set_bytes, 1)) + 1))
        sets = [make_set() for _ in range(nb)]
        for st in sets:
            call(st)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for st in sets:
                call(st)
        g.replay()
        reps = max(3, 200 // nb)
        us = time_graph(g, reps) * 1e3 / (reps * nb)
        if bound == "hbm":
            ach = alg_bytes / (us * 1e-6) / 1e9
            rows.append({"op": name, "us": round(us, 2), "bound": "hbm", "achieved": round(ach, 1),
                         "unit": "GB/s", "peak": hbm, "frac": round(ach / hbm, 4),
                         "algorithmic_bytes": int(alg_bytes), "rotating_sets": nb})
        else:
            ach = alg_flops / (us * 1e-6) / 1e12
            rows.append({"op": name, "us": round(us, 2), "bound": "tensor", "achieved": round(ach, 1),
                         "unit": "TFLOP/s", "peak": tc, "frac": round(ach / tc, 4),
                         "algorithmic_flops": int(alg_flops), "rotating_sets": nb})
        del sets
        torch.cuda.empty_cache()

    # a1 stats
    for (R, C) in [(25088, 64), (4096, 3072), (401408, 64)]:
        b = R * C * 2 + occ_b(R, C)
        measure(f"stats [{R},{C}]",
                lambda R=R, C=C: (act_like(R, C), sp.OccupancyBuffer(R, C)),
                lambda st, R=R, C=C: sp.sparoa_op_stats(ctx, st[0], (R, C), occ=st[1], host=False),
                b, alg_bytes=b)
    # a6 depthwise (MobileNetV2 layers), BN + ReLU6, output occupancy
    for (N, H, W, C, s) in [(32, 112, 112, 96, 2), (32, 56, 56, 144, 1)]:
        Ho, Wo = (H + 2 - 3) // s + 1, (W + 2 - 3) // s + 1
        w = (torch.randn(C, 3, 3, 1, device=dev, generator=gen) / 3).to(torch.bfloat16)
        bnp = torch.tensor(synth.identity_bn(C), device=dev)
        b = N * H * W * C * 2 + N * Ho * Wo * C * 2 + C * 9 * 2 + occ_b(N * Ho * Wo, C)
        measure(f"depthwise 3x3 s{s} [{N},{H},{W},{C}]",
                lambda N=N, H=H, W=W, C=C, Ho=Ho, Wo=Wo: (
                    act_like(N, H, W, C), torch.empty(N, Ho, Wo, C, dtype=torch.bfloat16, device=dev),
                    sp.OccupancyBuffer(N * Ho * Wo, C)),
                lambda st, w=w, s=s, C=C, bnp=bnp: sp.sparoa_conv2d(
                    ctx, st[0], w, st[1], stride=s, pad=1, groups=C, bn=bnp, act=sp.ACT_RELU6,
                    y_occ=st[2]),
                b, alg_bytes=b)
    # a7 pooling and stand-alone BN/activation
    b = 32 * 112 * 112 * 64 * 2 + 32 * 56 * 56 * 64 * 2 + occ_b(32 * 56 * 56, 64)
    measure("maxpool 3x3/2 [32,112,112,64]",
            lambda: (act_like(32, 112, 112, 64), torch.empty(32, 56, 56, 64, dtype=torch.bfloat16, device=dev),
                     sp.OccupancyBuffer(32 * 56 * 56, 64)),
            lambda st: sp.sparoa_maxpool2d(ctx, st[0], st[1], y_occ=st[2]), b, alg_bytes=b)
    b = 32 * 7 * 7 * 1280 * 2 + 32 * 1280 * 2 + occ_b(32, 1280)
    measure("avgpool global [32,7,7,1280]",
            lambda: (act_like(32, 7, 7, 1280), torch.empty(32, 1, 1, 1280, dtype=torch.bfloat16, device=dev),
                     sp.OccupancyBuffer(32, 1280)),
            lambda st: sp.sparoa_avgpool_global(ctx, st[0], st[1], y_occ=st[2]), b, alg_bytes=b)
    bnp64 = torch.tensor(synth.identity_bn(64), device=dev)
    b = 2 * 32 * 56 * 56 * 64 * 2 + occ_b(32 * 56 * 56, 64)
    measure("bn+relu [32,56,56,64]",
            lambda: (act_like(32, 56, 56, 64, zero_p=0.0), torch.empty(32, 56, 56, 64, dtype=torch.bfloat16, device=dev),
                     sp.OccupancyBuffer(32 * 56 * 56, 64)),
            lambda st: sp.sparoa_bn_act(ctx, st[0], st[1], bn=bnp64, act=sp.ACT_RELU, y_occ=st[2]),
            b, alg_bytes=b)
    # a4 zero-skip FC (column-sparse input: only occupied weight rows are read)
    d = synth.fc_layer(seed=0)
    M, K, N = d["M"], d["K"], d["N"]
    wfc = sp.bits_to_device(d["w"]).view(N, K)
    wkn = sp.bits_to_device(d["w_kn"]).view(K, N)
    x0 = sp.bits_to_device(d["x"]).view(M, K)
    kocc = int((x0.float().abs().sum(0) != 0).sum().item())
    b = kocc * N * 2 + M * K * 2 + M * N * 4
    measure(f"fc zero-skip [{M},{K}]x[{K},{N}] (occupied K {kocc})",
            lambda: (x0.clone(), torch.empty(M, N, dtype=torch.float32, device=dev)),
            lambda st: sp.sparoa_gemm(ctx, st[0], wfc, st[1], W_kn=wkn),
            M * K * 2 + M * N * 4, alg_bytes=b)
    # a5 dense GEMMs (MLP block) and the 3x3 conv
    for (M, K, N) in [(4096, 768, 3072), (4096, 3072, 768)]:
        w = (torch.randn(N, K, device=dev, generator=gen) / K ** 0.5).to(torch.bfloat16)
        measure(f"gemm dense [{M},{K}]x[{N},{K}]^T",
                lambda M=M, K=K, N=N: (act_like(M, K, zero_p=0.0), torch.empty(M, N, dtype=torch.bfloat16, device=dev),
                                       sp.OccupancyBuffer(M, K)),
                lambda st, w=w, M=M, K=K: (sp.sparoa_op_stats(ctx, st[0], (M, K), occ=st[2], host=False),
                                           sp.sparoa_gemm(ctx, st[0], w, st[1], x_occ=st[2],
                                                          thr=sp.thresholds(force_path=sp.PATH_DENSE))),
                M * K * 2 + M * N * 2, alg_flops=2.0 * M * K * N, bound="tensor")
    w3 = (torch.randn(64, 3, 3, 64, device=dev, generator=gen) / 24).to(torch.bfloat16)
    for force, tag in [(sp.PATH_DENSE, "dense"), (sp.PATH_SKIP, "zero-skip")]:
        measure(f"conv3x3 [32,56,56,64]->64 {tag}",
                lambda: (act_like(32, 56, 56, 64), torch.empty(32, 56, 56, 64, dtype=torch.bfloat16, device=dev),
                         sp.OccupancyBuffer(32 * 56 * 56, 64), sp.OccupancyBuffer(32 * 56 * 56, 64)),
                lambda st, force=force: (sp.sparoa_op_stats(ctx, st[0], (32, 56, 56, 64), occ=st[2], host=False),
                                         sp.sparoa_conv2d(ctx, st[0], w3, st[1], stride=1, pad=1, act=sp.ACT_RELU,
                                                          thr=sp.thresholds(force_path=force), x_occ=st[2],
                                                          y_occ=st[3])),
                2 * 32 * 56 * 56 * 64 * 2, alg_flops=2.0 * 32 * 56 * 56 * 64 * 64 * 9, bound="tensor")
    ctx.close()
    return {"metric": METRIC, "value": None, "unit": "per-op roofline", "n_gpus": world,
            "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "every kernel of the path at the workloads' shapes; the GEMM, FC and "
                                   "conv rows include their input's stats kernel",
                       "l2": "rotating sets totalling > 3 x 129 MB per graph"},
            "ops": rows}


def run_calibrate(args, rank, local_rank, world, peaks):
    """Per-operator threshold calibration (Sec. 3.3's ground-truth grid, on
    this GPU): forced dense vs forced zero-skip over rho x size x structure,
    the crossover table, then ResNet-18 (B=8) and MobileNetV2 (B=32) images/s
    under the default thresholds and under the fresh calibrated ones."""
    import torch

    from paper_2511_19457_gb300 import calibrate as cal
    from paper_2511_19457_gb300 import sparoa as sp
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    t0 = time.time()
    table = cal.calibrate(ctx, log=lambda e: print(json.dumps(
        {"kind": e["kind"], "shape": e["shape"], "structure": e["structure"], "s_thr": e["s_thr"],
         "dense_us": e["dense_us"], "skip_us": e["skip_us"]}), file=sys.stderr, flush=True))
    cal_s = time.time() - t0
    if args.calib_out:
        with open(args.calib_out, "w") as f:
            json.dump(table, f, indent=1)
    graphs = {}
    for name, batch in (("resnet18", 8), ("mobilenet_v2", 32)):
        res = {}
        for tag, thr in (("default", "default"), ("calibrated", table)):
            ms, recs = time_graph_workload(ctx, name, batch, 50, 5, thr)
            res[tag] = {"images_per_s": round(batch / (ms * 1e-3), 1), "ms": round(ms, 4),
                        "paths": "".join({0: "-", 1: "D", 2: "S", 3: "w"}.get(int(r.stats.path), "?")
                                         for r in recs)}
        graphs[f"{name}_b{batch}"] = res
    ctx.close()
    return {"metric": METRIC, "value": None, "unit": "crossover rho per operator", "n_gpus": world,
            "higher_is_better": False, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "threshold calibration: forced dense vs zero-skip per operator "
                                   "kind and size over rho x {unstructured, block}",
                       "seconds": round(cal_s, 1)},
            "crossover": cal.summary(table), "graphs": graphs}


def run_batching(args, rank, local_rank, world, peaks):
    """Dynamic batching (Algorithm 2) on the synthetic CNNs: every evaluated
    batch size is one CUDA-graph-captured sparoa_run_graph timed after an L2
    flush; M(B) is the graph walk's workspace plus the input."""
    import numpy as np
    import torch

    from paper_2511_19457_gb300 import batching as bt
    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    out = {}
    for name in ("resnet18", "mobilenet_v2"):
        ops, _, _ = getattr(synth, name)(batch=1)
        graph = sp.Graph(ops)
        gen = torch.Generator(device=dev).manual_seed(0)
        cache = {}

        def latency(B):
            if B in cache:
                return cache[B]
            x = torch.randn(B, 224, 224, 3, device=dev, generator=gen).to(torch.bfloat16)
            for _ in range(3):
                sp.sparoa_run_graph(ctx, graph, x)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                sp.sparoa_run_graph(ctx, graph, x)
            g.replay()
            ts = []
            for _ in range(20):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                g.replay()
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1) * 1e-3)
            del g, x
            cache[B] = float(np.median(ts))
            return cache[B]

        def memory(B):
            return sp.sparoa_graph_workspace(ctx, graph, (B, 224, 224, 3)) + B * 224 * 224 * 3 * 2

        # the input's operator-level characteristics, FLOP-weighted over conv / FC
        recs = sp.sparoa_run_graph(ctx, graph, torch.randn(8, 224, 224, 3, device=dev, generator=gen)
                                   .to(torch.bfloat16), records=True)
        fl = np.array([r.stats.flops for r in recs], dtype=np.float64)
        rho = float((fl * np.array([r.stats.sparsity for r in recs])).sum() / fl.sum())
        fpb = float((fl * np.array([r.stats.flops_per_byte for r in recs])).sum() / fl.sum())
        tr = bt.dynamic_batch(latency, memory, 1, sparsity=rho, intensity=fpb, s_thr=0.5, c_thr=None,
                              mem_max=32 * 2 ** 30, t_realtime=2e-3, b_max=256)
        out[name] = {"input_sparsity": round(rho, 4), "input_flops_per_byte": round(fpb, 1),
                     **tr.as_dict()}
    ctx.close()
    return {"metric": METRIC, "value": None, "unit": "batch size", "n_gpus": world,
            "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "Algorithm 2 dynamic batching over sparoa_run_graph",
                       "constraints": {"mem_max_gib": 32, "t_realtime_ms": 2.0, "s_thr": 0.5,
                                       "c_thr": None, "B0": 1, "b_max": 256},
                       "l2": "flushed by a 256 MB write before every timed replay"},
            "graphs": out}


def run_split(args, rank, local_rank, world, peaks):
    """Split execution on a batch of mixed sparsity: the MLP down projection
    h [4096, 3072] x W2 [768, 3072]^T whose first `frac_sparse` of tokens carry
    block-structured zeros at rho 0.9 and the rest none.  Dense, zero-skip and
    split (rows [0, xi M) zero-skip, the rest dense, two streams) per call,
    CUDA-graph replays over rotating sets larger than L2."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    gen = torch.Generator(device=dev).manual_seed(0)
    M, K, N = 4096, 3072, 768
    W = (torch.randn(N, K, device=dev, generator=gen) / K ** 0.5).to(torch.bfloat16)
    nb = 6
    rows = []
    for frac_sparse in (0.25, 0.5, 0.75):
        ms = int(M * frac_sparse)
        xs = []
        for _ in range(nb):
            h = synth.structured_activation((M, K), 0.9, "block", gen, dev)
            h[ms:] = (torch.randn(M - ms, K, device=dev, generator=gen).abs() + 1e-3).to(torch.bfloat16)
            xs.append(h)
        ys = [torch.empty(M, N, dtype=torch.bfloat16, device=dev) for _ in range(nb)]
        occ = [sp.OccupancyBuffer(M, K) for _ in range(nb)]
        for j in range(nb):
            sp.sparoa_op_stats(ctx, xs[j], (M, K), occ=occ[j], host=False)
        calls = {"dense": lambda j: sp.sparoa_gemm(ctx, xs[j], W, ys[j], thr=sp.thresholds(force_path=1),
                                                   x_occ=occ[j]),
                 "zero-skip": lambda j: sp.sparoa_gemm(ctx, xs[j], W, ys[j],
                                                       thr=sp.thresholds(force_path=2), x_occ=occ[j])}
        for xi in (0.25, 0.5, 0.75):
            calls[f"split xi={xi}"] = lambda j, xi=xi: sp.sparoa_gemm_split(ctx, xs[j], W, ys[j], xi,
                                                                             x_occ=occ[j])
        res = {}
        for tag, call in calls.items():
            for j in range(nb):
                call(j)
            torch.cuda.synchronize()
            g = graph_of(call, nb)
            g.replay()
            res[tag] = round(time_graph(g, 20) * 1e3 / (20 * nb), 2)
            del g
        rows.append({"sparse_token_fraction": frac_sparse, "us_per_call": res,
                     "best": min(res, key=res.get)})
        del xs, ys, occ
        torch.cuda.empty_cache()
    ctx.close()
    return {"metric": METRIC, "value": None, "unit": "us per call", "n_gpus": world,
            "higher_is_better": False, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "split execution: MLP down projection [4096,3072]x[768,3072]^T, "
                                   "a fraction of tokens block-sparse (rho 0.9), the rest dense",
                       "l2": "rotating sets of 6 x (24 MB in + 6 MB out) > 129 MB"},
            "rows": rows}


def run_profile(args, rank, local_rank, world, peaks):
    """One operator at a workload shape, called 4 times on the same inputs (no
    CUDA graph): the fixed launch sequence that the committed ncu summaries
    capture (e.g. ``-k regex:conv3 -s 3 -c 1`` takes the 4th launch).  Inputs
    larger than L2 are the bench's shapes; the 4th call finds them partly in
    L2 (a capture's DRAM bytes are read against that)."""
    import torch

    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    ctx = sp.Context(local_rank)
    gen = torch.Generator(device=dev).manual_seed(0)

    def act(*shape, zero_p=0.5):
        v = torch.randn(*shape, device=dev, generator=gen).abs()
        v[torch.rand(*shape, device=dev, generator=gen) < zero_p] = 0.0
        return v.to(torch.bfloat16)

    op = args.op
    if op == "conv_cfg2":  # the default bench step: stats + dispatch + 3x3 conv, BN + ReLU
        d = synth.conv_layer(seed=0)
        x = sp.bits_to_device(d["x"]).view(8, 56, 56, 64)
        w = sp.bits_to_device(d["w"]).view(64, 3, 3, 64)
        bn = torch.from_numpy(d["bn"]).to(dev)
        y = torch.empty(8, 56, 56, 64, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(8 * 56 * 56, 64)
        call = lambda: sp.sparoa_conv2d(ctx, x, w, y, stride=1, pad=1, bn=bn, act=sp.ACT_RELU, y_occ=yo)
    elif op == "fc_cfg1":
        d = synth.fc_layer(seed=0)
        x = sp.bits_to_device(d["x"]).view(64, 512)
        w = sp.bits_to_device(d["w"]).view(512, 512)
        wkn = sp.bits_to_device(d["w_kn"]).view(512, 512)
        y = torch.empty(64, 512, dtype=torch.float32, device=dev)
        call = lambda: sp.sparoa_gemm(ctx, x, w, y, W_kn=wkn)
    elif op in ("gemm_dense_mlp", "gemm_skip_mlp_block32"):
        wts = synth.mlp_weights(seed=0)
        w2 = sp.bits_to_device(wts["w2"]).view(768, 3072)
        h = sp.bits_to_device(synth.mlp_hidden(4096, 0.5, "block32", seed=1)).view(4096, 3072)
        y = torch.empty(4096, 768, dtype=torch.bfloat16, device=dev)
        force = 1 if op == "gemm_dense_mlp" else 2
        call = lambda: sp.sparoa_gemm(ctx, h, w2, y, thr=sp.thresholds(force_path=force))
    elif op in ("dw3_s2", "dw3_s1"):
        N, H, W, C, s_ = (32, 112, 112, 96, 2) if op == "dw3_s2" else (32, 56, 56, 144, 1)
        Ho, Wo = (H + 2 - 3) // s_ + 1, (W + 2 - 3) // s_ + 1
        x = act(N, H, W, C)
        w = (torch.randn(C, 3, 3, 1, device=dev, generator=gen) / 3).to(torch.bfloat16)
        bnp = torch.tensor(synth.identity_bn(C), device=dev)
        y = torch.empty(N, Ho, Wo, C, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(N * Ho * Wo, C)
        call = lambda: sp.sparoa_conv2d(ctx, x, w, y, stride=s_, pad=1, groups=C, bn=bnp, act=sp.ACT_RELU6, y_occ=yo)
    elif op == "maxpool":
        x = act(32, 112, 112, 64)
        y = torch.empty(32, 56, 56, 64, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(32 * 56 * 56, 64)
        call = lambda: sp.sparoa_maxpool2d(ctx, x, y, y_occ=yo)
    elif op == "bn_act":
        x = act(32, 56, 56, 64, zero_p=0.0)
        bnp = torch.tensor(synth.identity_bn(64), device=dev)
        y = torch.empty(32, 56, 56, 64, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(32 * 56 * 56, 64)
        call = lambda: sp.sparoa_bn_act(ctx, x, y, bn=bnp, act=sp.ACT_RELU, y_occ=yo)
    elif op == "conv1x1_expand":  # MobileNetV2's first expansion at batch 32, BN + ReLU6
        x = act(32, 112, 112, 16)
        w = (torch.randn(96, 1, 1, 16, device=dev, generator=gen) / 4).to(torch.bfloat16)
        bnp = torch.tensor(synth.identity_bn(96), device=dev)
        y = torch.empty(32, 112, 112, 96, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(32 * 112 * 112, 96)
        call = lambda: sp.sparoa_conv2d(ctx, x, w, y, bn=bnp, act=sp.ACT_RELU6, y_occ=yo)
    elif op == "stem7x7":  # ResNet-18's stem at batch 32: im2col rows, then a GEMM; BN + ReLU
        x = act(32, 224, 224, 3, zero_p=0.0)
        w = (torch.randn(64, 7, 7, 3, device=dev, generator=gen) / 12).to(torch.bfloat16)
        bnp = torch.tensor(synth.identity_bn(64), device=dev)
        y = torch.empty(32, 112, 112, 64, dtype=torch.bfloat16, device=dev)
        yo = sp.OccupancyBuffer(32 * 112 * 112, 64)
        call = lambda: sp.sparoa_conv2d(ctx, x, w, y, stride=2, pad=3, bn=bnp, act=sp.ACT_RELU, y_occ=yo)
    elif op == "stats_large":
        x = act(401408, 64)
        oc = sp.OccupancyBuffer(401408, 64)
        call = lambda: sp.sparoa_op_stats(ctx, x, (401408, 64), occ=oc, host=False)
    else:
        raise SystemExit(f"profile: unknown op {op}")
    t0 = time.perf_counter()
    for _ in range(4):
        call()
    torch.cuda.synchronize()
    ctx.close()
    return {"workload": "profile", "op": op, "calls": 4, "seconds": time.perf_counter() - t0}


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    rank, local_rank, world = dist_env()
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    peaks = measured_peaks()
    if args.workload == "conv":
        line = run_conv(args, rank, local_rank, world, peaks)
        if world == 1 and not args.no_extras:
            import torch

            from paper_2511_19457_gb300 import sparoa as sp
            ctx = sp.Context(local_rank)
            line["other_configs"] = other_configs(ctx, torch.device("cuda", local_rank), peaks)
            ctx.close()
        if rank == 0 and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline_conv()
            if "other_configs" in line:
                line["cpu_baseline"]["oracle_rule_check"] = oracle_rule_check(line["other_configs"])
        if "other_configs" in line:
            for rec in line["other_configs"].get("graphs", {}).values():
                if isinstance(rec, dict):
                    rec.pop("decisions", None)
    elif args.workload in ("resnet18", "mobilenet_v2", "vit_b16"):
        line = run_graph_workload(args, rank, local_rank, world, peaks, args.workload)
    elif args.workload == "fc":
        line = run_fc(args, rank, local_rank, world, peaks)
    elif args.workload == "mlp_sweep":
        line = run_mlp_sweep(args, rank, local_rank, world, peaks)
    elif args.workload == "ops":
        line = run_ops(args, rank, local_rank, world, peaks)
    elif args.workload == "calibrate":
        line = run_calibrate(args, rank, local_rank, world, peaks)
    elif args.workload == "batching":
        line = run_batching(args, rank, local_rank, world, peaks)
    elif args.workload == "split":
        line = run_split(args, rank, local_rank, world, peaks)
    elif args.workload == "profile":
        line = run_profile(args, rank, local_rank, world, peaks)
    else:
        raise SystemExit(f"workload {args.workload} is not wired into bench.py")
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

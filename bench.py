#!/usr/bin/env python
"""Benchmark of the Chameleon format-adaptive quantized linear path on GB300.

Headline workload: every linear of a PixArt-alpha-architecture DiT (28 blocks, hidden 1152, MLP
4608, 4096 image + 120 caption tokens per sample, batch 2: 282 linears per sampler step) over a
20-step sampler, W4A8.  One benchmark step is one pass of the whole hot path: per-channel
weight-format selection over the 4-bit palette {INT4-asym, NF4, E2M1, MXINT4, MXFP4} and the pack
of all 282 layers, then 20 sampler steps (t = 999 - 50 i) in which every linear quantizes its input
with each sample's own range (Alg. 3) in the format its (layer, timestep-bucket) table entry names
and multiplies (fp32 outputs).  Linears that read the same tensor run as one GEMM with their
weights stacked along N -- each block's q, k, v, and the cross-attention k, v of all 28 blocks
(they all read the caption tokens): 171 GEMMs per sampler step, the same per-channel formats,
activation codes and outputs.  Random-init weights, seeded synthetic activations.

Sub-objects: the SDXL-UNet W8A8 projection step (static calibrated scales, Alg. 2), the GEMM for
every activation x weight format, the public quantizer per format and shape, selection and pack,
the other workloads' shapes (SDXL-UNet W4A8, SDXL-Turbo W4A16 batch sweep) and the group-wise DiT
fork.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on a bounded sample of the
same workload instead.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

if "--oracle-sample" not in sys.argv:
    # the oracle's timed legs pick their BLAS thread count in a child process (cpu_baseline)
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "mixed-format linear TFLOP/s & % tensor peak; act-quant HBM GB/s"
WORKLOAD = ("PixArt-alpha DiT, all 282 linears (28 blocks + caption projection), batch 2 x (4096 + 120) tokens, "
            "W4A8, 20-step sampler, per-(layer, bucket) activation formats, per-sample dynamic scales")
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FP8_OVER_BF16 = 2.0  # nominal dense FP8 / bf16 tensor rate (4.5 / 2.25 PFLOP/s per GPU)
# the 4-bit palette of the DiT and few-step forks (Sec. 3.5): INT4-asym, NF4, E2M1, MXINT4, MXFP4
W4_PALETTE = (1 << 4) | (1 << 5) | (1 << 6) | (1 << 7) | (1 << 8)
# dram__bytes_read.sum + dram__bytes_write.sum of one launch of the dominant kernel from an ncu
# capture (profiles/), with the launch it was and that launch's algorithmic bytes.  None whenever
# the kernel has changed since the capture.  Captured: k_gemm_ts_f8<192, 1, 0> on
# `--case gemm-pixart-qkv`, one launch of the headline's stacked q/k/v GEMM at full size.
GEMM_TRAFFIC_PER_LAUNCH = {"bytes": 132.8e6, "launch": "8192 x 1152 x 3456 (PixArt-alpha q/k/v stacked, E4M3, "
                                                     "per-sample scales, fp32 Y)", "algorithmic_bytes": 143.5e6}


def traffic_fields(t=GEMM_TRAFFIC_PER_LAUNCH):
    """roofline.traffic (DRAM bytes of one captured launch, or None) and what that launch was."""
    if not t:
        return {"traffic": None}
    return {"traffic": t["bytes"], "traffic_launch": t["launch"], "traffic_algorithmic_bytes": t["algorithmic_bytes"]}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return PEAKS_FALLBACK, "fallback"


# ------------------------------------------------------------------ clocks during the timed region
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]
        return False

    def summary(self):
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ replicas (N > 1)
def max_over_ranks(ms, device=None):
    """The slowest rank's time: every rank gets the maximum (the job ends with its last rank)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tflops(flops_step, steps, world, max_ms):
    """Whole-job throughput: every rank runs the full step (weak scaling, independent replicas)."""
    return world * flops_step * steps / (max_ms * 1e-3) / 1e12


def layer_flops(M, K, N):
    return 2.0 * M * K * N


def graph_timer(torch, reps=20):
    """fn -> milliseconds per call: `reps` calls captured in one CUDA graph, replayed once warm and
    then timed between two events on the current stream (the launches alone, back to back)."""
    def timed(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(reps):
                fn()
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps
    return timed


# ------------------------------------------------------------------ the PixArt-alpha inputs
def pixart_host_inputs(workers):
    """Weights and biases of the 282 linears and the 7 input tensors at the 10 timestep buckets,
    generated by the seeded workload module in a pool of `workers` spawned processes (started
    before this process touches the GPU).  Returns (weights, biases, inputs[(key, bucket)])."""
    import concurrent.futures
    import multiprocessing
    from paper_2609_33496_gb300 import workloads as WL
    n = len(WL.pixart_model_linears())
    keys = sorted(WL.PIXART_INPUTS)
    ctx = multiprocessing.get_context("spawn")
    with concurrent.futures.ProcessPoolExecutor(max_workers=workers, mp_context=ctx) as ex:
        xf = {(k, b): ex.submit(WL.pixart_model_input, k, b) for k in keys for b in range(10)}
        wf = [ex.submit(WL.pixart_model_weights, i) for i in range(n)]
        W, bias = zip(*[f.result() for f in wf])
        X = {kb: f.result() for kb, f in xf.items()}
    return list(W), list(bias), X


def pixart_calibrate(cl, Xd):
    """Alg. 1 on the synthetic activations: per input tensor and bucket, the power sums on the GPU,
    kappa, the SNR at the bucket midpoint on the linear schedule (PixArt-alpha), Route -> the
    activation format.  Returns lut[(key, bucket)] (linears reading the same tensor share it)."""
    snr = cl.snr(cl.SCHEDULE_LINEAR, 1000)
    lut = {}
    for (key, b), x in Xd.items():
        sums = cl.act_moments(x).cpu().numpy()
        lut[(key, b)] = int(cl.route(cl.kurtosis(sums[:5]), snr[b * 100 + 50], False))
    return lut


def pixart_headline(args, torch, cl, WL, host, device, world, st):
    """The headline step (module docstring).  Returns the result fields and what the e2e leg and
    the sub-objects reuse."""
    import torch.distributed as dist
    Wn, bn, Xn = host
    n_linears = len(WL.pixart_model_linears())
    linears = WL.pixart_model_gemms()   # (names, M, K, N, input, indices): q/k/v and cross k/v stacked
    n = len(linears)
    W = [torch.from_numpy(np.concatenate([Wn[i] for i in ix])).to(device) for (_, M, K, N, _, ix) in linears]
    bias = [torch.from_numpy(np.concatenate([bn[i] for i in ix])).to(device) for (_, M, K, N, _, ix) in linears]
    X = {kb: torch.from_numpy(x).to(device) for kb, x in Xn.items()}
    lut = pixart_calibrate(cl, X)
    ts = WL.PIXART_SAMPLER_T[:args.sampler_steps]
    buckets = [cl.bucket(t) for t in ts]
    stream = torch.cuda.current_stream()

    # a5: selection into one format buffer; the packed layout needs the formats on the host (the
    # palette spans both MMA classes), so the step copies them back once for all layers
    offs = np.cumsum([0] + [N for (_, M, K, N, _, _) in linears])
    fmt_all = torch.empty(int(offs[-1]), dtype=torch.uint8, device=device)
    fmt_host = torch.empty(int(offs[-1]), dtype=torch.uint8).pin_memory()

    def select_layers():
        for i in range(n):
            cl.select_weight_formats(W[i], W4_PALETTE, fmt_out=fmt_all[offs[i]:offs[i + 1]])

    select_layers()
    fmt_host.copy_(fmt_all, non_blocking=True)
    torch.cuda.synchronize()
    f_ref = fmt_host.numpy().copy()
    descs = [cl.pack_plan(N, K, f_ref[offs[i]:offs[i + 1]]) for i, (_, M, K, N, _, _) in enumerate(linears)]
    blobs = [torch.empty(d.bytes, dtype=torch.uint8, device=device) for d in descs]

    def pack_layers():
        for i in range(n):
            cl.pack_weights(W[i], fmt_all[offs[i]:offs[i + 1]], descs[i], dev_status=st, blob=blobs[i])

    # the 171 selections and the 171 packs as two CUDA graphs (their arguments are the same every
    # step; the plans are checked against the formats each step selects)
    pack_layers()
    torch.cuda.synchronize()
    g_select, g_pack = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_select):
        select_layers()
    with torch.cuda.graph(g_pack):
        pack_layers()

    def select_all():
        g_select.replay()
        fmt_host.copy_(fmt_all, non_blocking=True)

    def plan_and_pack():
        """a6 for every layer, from the plans of the formats just selected (the same plans every
        step: the selection is deterministic; the step checks it)."""
        torch.cuda.current_stream().synchronize()
        f = fmt_host.numpy()
        if not np.array_equal(f, f_ref):
            raise RuntimeError("the selected formats changed between steps")
        g_pack.replay()

    acts = sorted(set(lut.values()))
    ws = torch.empty(max(cl.linear_workspace_size(M, descs[i], a) for i, (_, M, K, N, _, _) in enumerate(linears)
                         for a in acts), dtype=torch.uint8, device=device)
    # one output buffer per kind of GEMM (the blocks run in order; the benchmark keeps no model state)
    kind = [names[0].split(".", 1)[1] if names[0].startswith("block") else names[0] for (names, *_r) in linears]
    Ybuf = {}
    for k, (names, M, K, N, _, _) in zip(kind, linears):
        if k not in Ybuf:
            Ybuf[k] = torch.empty((M, N), dtype=torch.float32, device=device)
    Y = [Ybuf[k] for k in kind]

    def sampler(parts="qg"):
        """20 sampler steps: per linear the quantizer with the two samples' own scales (Alg. 3) in
        F[l, b(t)] ("q") and the GEMM ("g")."""
        for b in buckets:
            for i, (names, M, K, N, key, _) in enumerate(linears):
                af = lut[(key, b)]
                x = X[(key, b)]
                if "q" in parts:
                    cl.linear_prepare_groups(x, descs[i], af, 2, ws, st)
                if "g" in parts:
                    cl.linear_gemm_ex(x, descs[i], blobs[i], af, 2, bias[i], Y[i], ws, st)

    def step(graphs):
        select_all()
        plan_and_pack()
        graphs["qg"].replay()

    for _ in range(2):
        sampler()
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    graphs = {}
    for key in ("qg", "q", "g"):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            sampler(key)
        graphs[key] = g
    for _ in range(args.warmup):
        step(graphs)
    torch.cuda.synchronize()

    # launches per benchmark step: per layer the selection and the two pack kernels (slot plan and
    # pack: the palette spans both MMA classes); per linear the quantizer (range +
    # encode for the per-tensor formats, one launch for MX) and the GEMM (+ the split-K reduction)
    per_linear = {}
    for b in buckets:
        for i, (_, M, K, N, key, _) in enumerate(linears):
            k = (i, lut[(key, b)])
            if k not in per_linear:
                per_linear[k] = sum(cl.linear_launches(M, descs[i], lut[(key, b)], 2))
    launches = 3 * n + sum(per_linear[(i, lut[(key, b)])] for b in buckets
                           for i, (_, M, K, N, key, _) in enumerate(linears))
    flops_step = len(buckets) * sum(layer_flops(M, K, N) for (_, M, K, N, _, _) in linears)

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(device.index) as clk:
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        torch.cuda.nvtx.range_push("pixart_step")   # a profiler can take exactly the timed steps
        for _ in range(args.steps):
            step(graphs)
        torch.cuda.nvtx.range_pop()
        t1.record(stream)
        torch.cuda.synchronize()
        # kernel classes over the same period: the sampler's GEMMs alone and its quantizers alone
        # (graph replays, once per timed step), and the selection + pack (two graph replays)
        cls = {}
        for key in ("g", "q"):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(args.steps):
                graphs[key].replay()
            e1.record(stream)
            torch.cuda.synchronize()
            cls[key] = e0.elapsed_time(e1) / args.steps
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            select_all()
            plan_and_pack()
        e1.record(stream)
        torch.cuda.synchronize()
        cls["w"] = e0.elapsed_time(e1) / args.steps
    if world > 1:
        dist.barrier()
    elapsed_ms = t0.elapsed_time(t1)
    if world > 1:
        elapsed_ms = max_over_ranks(elapsed_ms, device)
    assert int(st.item()) == 0, "device status %d" % int(st.item())

    # per-layer class split of the flops (FP8 MMAs on class-0 tiles, fp16 MMAs on NF4 tiles) and
    # the quantizer's algorithmic bytes (2 B read + 1 B code per element, + 1/32 B for MX formats)
    fl8 = fl16 = 0.0
    qbytes = 0.0
    for b in buckets:
        for i, (_, M, K, N, key, _) in enumerate(linears):
            d, af = descs[i], lut[(key, b)]
            fl = layer_flops(M, K, N)
            share8 = d.n_class[0] / N if (af in (1, 2, 3)) else 0.0
            fl8 += fl * share8
            fl16 += fl * (1 - share8)
            qbytes += M * K * (3 + (1 / 32 if af in (3, 4) else 0))
    hist = np.bincount(f_ref, minlength=9)
    return {
        "value_tflops": job_tflops(flops_step, args.steps, world, elapsed_ms), "elapsed_ms": elapsed_ms,
        "flops_step": flops_step, "fl8": fl8, "fl16": fl16, "qbytes": qbytes, "classes_ms": cls,
        "launches": launches, "clocks": clk.summary(), "linears": linears, "lut": lut, "buckets": buckets,
        "descs": descs, "weight_formats": {int(f): int(c) for f, c in enumerate(hist) if c},
        "acts": acts, "n_linears": n_linears,
    }


# ------------------------------------------------------------------ SDXL-UNet W8A8 projections (config 2)
def sdxl_step(args, torch, cl, WL, device, st, pk):
    """The SDXL-UNet attention/FFN projections at batch 2 (q/k/v/out 8192x640x640 x4,
    2048x1280x1280 x4, GEGLU-in 2048x1280x10240, FF-out 2048x5120x1280), W8A8, over the 10
    timestep buckets: fused selection + pack of the 10 layers (the W8 palette is one MMA class, so
    the whole step is one CUDA graph), then per (bucket, layer) the quantizer with the static
    calibrated (S, Z)[l, b] of the UNet path (Alg. 2) in the LUT's format and the GEMM."""
    layers = WL.SDXL_PROJ_LAYERS
    nb = 10
    W, bias, X = [], [], []
    for li in range(len(layers)):
        w, b = WL.sdxl_layer_weights(li)
        W.append(torch.from_numpy(w).to(device))
        bias.append(torch.from_numpy(b).to(device))
        X.append([torch.from_numpy(WL.sdxl_layer_activation(li, bk)).to(device) for bk in range(nb)])
    snr = cl.snr(cl.SCHEDULE_SCALED_LINEAR, 1000)
    lut = np.zeros((len(layers), nb), dtype=np.int64)
    qp = [[None] * nb for _ in layers]
    sse = np.zeros((len(layers), nb, 5))
    for li in range(len(layers)):
        for bk in range(nb):
            sums = cl.act_moments(X[li][bk]).cpu().numpy()
            lut[li, bk] = cl.route(cl.kurtosis(sums[:5]), snr[bk * 100 + 50], False)
            if lut[li, bk] <= 2:
                qp[li][bk] = cl.scale_zp(int(lut[li, bk]), float(sums[5]), float(sums[6]))
            sse[li, bk] = cl.act_format_sse(X[li][bk])[0].cpu().numpy()
    descs = [cl.pack_plan_palette(N, K, cl.PALETTE_W8) for (_, M, K, N) in layers]
    blobs = [torch.empty(d.bytes, dtype=torch.uint8, device=device) for d in descs]
    offs = np.cumsum([0] + [N for (_, M, K, N) in layers])
    fmt_all = torch.empty(int(offs[-1]), dtype=torch.uint8, device=device)
    Y = [torch.empty((M, N), dtype=torch.float32, device=device) for (_, M, K, N) in layers]
    ws = [torch.empty(max(cl.linear_workspace_size(M, descs[li], f) for f in range(6)), dtype=torch.uint8,
                      device=device) for li, (_, M, K, N) in enumerate(layers)]

    def run(parts="wqg"):
        if "w" in parts:
            for li in range(len(layers)):
                cl.select_pack_palette(W[li], cl.PALETTE_W8, descs[li], fmt_out=fmt_all[offs[li]:offs[li + 1]],
                                       blob=blobs[li], dev_status=st)
        for bk in range(nb):
            for li in range(len(layers)):
                f = int(lut[li, bk])
                if "q" in parts:
                    cl.linear_prepare_static(X[li][bk], descs[li], f, qp[li][bk], ws[li], st)
                if "g" in parts:
                    cl.linear_gemm(X[li][bk], descs[li], blobs[li], f, bias[li], Y[li], ws[li], st)

    for _ in range(args.warmup):
        run()
    torch.cuda.synchronize()
    graphs = {}
    for key in ("wqg", "g", "q"):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            run(key)
        graphs[key] = g
    graphs["wqg"].replay()
    torch.cuda.synchronize()
    ms = {}
    for key in ("wqg", "g", "q"):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            graphs[key].replay()
        e1.record()
        torch.cuda.synchronize()
        ms[key] = e0.elapsed_time(e1) / args.steps
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    flops = nb * sum(layer_flops(M, K, N) for (_, M, K, N) in layers)
    peak16 = pk["bf16_tflops"]
    qbytes = nb * sum(M * K * 4 for (_, M, K, N) in layers)   # 2 B read + 2 B fp16 operand per element
    return {"workload": "SDXL-UNet attention/FFN projections, W8A8, batch 2 (CFG), 10 timestep buckets, static "
                        "calibrated scales (Alg. 2)",
            "tflops": round(flops / (ms["wqg"] * 1e-3) / 1e12, 1), "ms_per_step": round(ms["wqg"], 3),
            "gemm_tflops": round(flops / (ms["g"] * 1e-3) / 1e12, 1),
            "gemm_frac_bf16_burst": round(flops / (ms["g"] * 1e-3) / 1e12 / peak16, 4),
            "quant_ms": round(ms["q"], 3), "quant_gbs": round(qbytes / (ms["q"] * 1e-3) / 1e9, 1),
            "lut": [[int(v) for v in row] for row in lut],
            "calibration": route_vs_argmin(cl, lut, sse)}


def route_vs_argmin(cl, lut, sse):
    """How the kappa / SNR route (Sec. 3.3) compares with the exhaustive argmin of Eq.
    format-argmin on the same calibration tensors."""
    best = np.array([[cl.act_format_argmin(sse[i, j]) for j in range(sse.shape[1])] for i in range(sse.shape[0])])
    picked = np.take_along_axis(sse, lut[..., None], axis=2)[..., 0]
    opt = np.take_along_axis(sse, best[..., None], axis=2)[..., 0]
    ratio = picked / np.maximum(opt, 1e-300)
    best3 = np.array([[cl.act_format_argmin(list(sse[i, j, :3]) + [np.inf, np.inf]) for j in range(sse.shape[1])]
                      for i in range(sse.shape[0])])
    opt3 = np.take_along_axis(sse, best3[..., None], axis=2)[..., 0]
    ratio3 = picked / np.maximum(opt3, 1e-300)
    return {"agree": round(float((best == lut).mean()), 3),
            "sse_ratio_route_over_argmin": {"median": round(float(np.median(ratio)), 3),
                                            "max": round(float(ratio.max()), 3)},
            "agree_per_tensor_formats": round(float((best3 == lut).mean()), 3),
            "sse_ratio_route_over_per_tensor_argmin": {"median": round(float(np.median(ratio3)), 3),
                                                       "max": round(float(ratio3.max()), 3)},
            "argmin_formats": {int(f): int(c) for f, c in zip(*np.unique(best, return_counts=True))},
            "route_formats": {int(f): int(c) for f, c in zip(*np.unique(lut, return_counts=True))}}


# ------------------------------------------------------------------ per-variant tables
def gemm_matrix(torch, cl, WL, st, p16, p8, hbm, shape=(8192, 1152, 4608)):
    """The GEMM for every activation format x weight format on one shape (PixArt-alpha fc1 by
    default): 5 x 9 W8A8 / W4A8 pairs (every channel in one format) and W4A16 x the 6 4-bit
    formats, each as 20 graph-captured launches.  Per pair: TFLOP/s, which MMA kind runs it, and
    the fraction of its roofline max(flops / P, algorithmic bytes / HBM) with P the kind's peak."""
    M, K, N = shape
    g = np.random.default_rng(20264000)
    dev = torch.device("cuda", torch.cuda.current_device())
    X = torch.from_numpy(WL.to_fp16(g.standard_t(7, (M, K)) * np.exp(0.1 * g.standard_normal(K))[None, :])).to(dev)
    W = torch.from_numpy(WL.weight_mix_rows(g, N, K)).to(dev)
    Y = torch.empty((M, N), dtype=torch.float32, device=dev)
    timed = graph_timer(torch)
    rows = []
    fl = layer_flops(M, K, N)
    for wf in range(9):
        fmt_h = np.full(N, wf, np.uint8)
        d = cl.pack_plan(N, K, fmt_h)
        blob, _ = cl.pack_weights(W, torch.from_numpy(fmt_h).to(dev), d, dev_status=st)
        bits = 8 if wf <= 2 else 4
        for af in range(6):
            if af == 5 and bits == 8:
                continue
            ws = torch.empty(cl.linear_workspace_size(M, d, af), dtype=torch.uint8, device=dev)
            if af != 5:
                cl.linear_prepare(X, d, af, ws, st)
            t = timed(lambda: cl.linear_gemm(X, d, blob, af, None, Y, ws, st)) * 1e-3
            fp8 = bits == 4 and af in (1, 2, 3) and wf not in (5,)
            peak = p8 if fp8 else p16
            a_bytes = M * K * (2 if af == 5 else 1) + (M * K / 32 if af in (3, 4) else 0)
            byts = a_bytes + N * K * bits / 8 + (N * K / 32 if wf in (2, 7, 8) else 5 * N) + 4 * N + 4 * M * N
            t_roof = max(fl / peak, byts / hbm)
            rows.append({"act_fmt": af, "w_fmt": wf, "us": round(t * 1e6, 2), "tflops": round(fl / t / 1e12, 1),
                         "mma": "kind::mxf8f6f4" if fp8 else "kind::f16",
                         "peak_tflops": round(peak / 1e12, 1), "frac_roofline": round(t_roof / t, 4)})
            del ws
    # the same weights with per-channel selection over the 4-bit palette (both MMA classes in one
    # launch), E4M3 activations
    fmt, _ = cl.select_weight_formats(W, W4_PALETTE)
    d = cl.pack_plan(N, K, fmt.cpu().numpy())
    blob, _ = cl.pack_weights(W, fmt, d, dev_status=st)
    ws = torch.empty(cl.linear_workspace_size(M, d, 1), dtype=torch.uint8, device=dev)
    cl.linear_prepare(X, d, 1, ws, st)
    t = timed(lambda: cl.linear_gemm(X, d, blob, 1, None, Y, ws, st)) * 1e-3
    f8 = d.n_class[0] / N
    t_roof = fl * f8 / p8 + fl * (1 - f8) / p16
    selected = {"act_fmt": 1, "w_fmt": "selected", "channels_fp8": int(d.n_class[0]), "channels_nf4": int(d.n_class[1]),
                "us": round(t * 1e6, 2), "tflops": round(fl / t / 1e12, 1), "frac_roofline": round(t_roof / t, 4)}
    del ws
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return {"shape": [M, K, N], "reps": 20, "rows": rows, "selected": selected,
            "note": "act_fmt 0 INT8-asym, 1 E4M3, 2 E5M2, 3 MXFP8, 4 MXINT8, 5 fp16; w_fmt 0 INT8-sym, 1 INT8-asym, "
                    "2 MXINT8, 3 INT4-sym, 4 INT4-asym, 5 NF4, 6 E2M1, 7 MXINT4, 8 MXFP4"}


def quant_tables(torch, cl, WL, hbm):
    """The public quantizer (chameleon_act_quant: 1-byte codes, E8M0 exponents for MX, the range
    pass for per-tensor formats) per activation format: on one 8192x4608 tensor (PixArt-alpha fc2's
    input), on 8192x1152 tensors (its hidden states), on each of the 22 distinct GEMM inputs of an
    SDXL-UNet step, and over those 22 in aggregate.  Algorithmic bytes: 2 B read + 1 B code per element (+ 1/32 B for MX).  The tensors
    are larger than L2 or, where not, their launches are back to back on distinct tensors."""
    dev = torch.device("cuda", torch.cuda.current_device())
    timed = graph_timer(torch, reps=10)
    g = np.random.default_rng(20265000)
    out = {"big": [], "unet_step": [], "unet_aggregate": []}

    def one(M, K, fmt, X):
        qb, wb = cl.act_quant_size(M, K, fmt)
        q = torch.empty(qb, dtype=torch.uint8, device=dev)
        ws = torch.empty(max(wb, 256), dtype=torch.uint8, device=dev)
        stq = torch.zeros(1, dtype=torch.int32, device=dev)
        t = timed(lambda: cl.act_quant(X, fmt, qact=q, ws=ws, dev_status=stq)) * 1e-3
        byts = M * K * (3 + (1 / 32 if fmt >= 3 else 0))
        return t, byts

    Xb = torch.from_numpy(WL.to_fp16(g.standard_t(5, (8192, 4608)))).to(dev)
    for fmt in range(5):
        t, byts = one(8192, 4608, fmt, Xb)
        out["big"].append({"fmt": fmt, "M": 8192, "K": 4608, "us": round(t * 1e6, 2),
                           "gbs": round(byts / t / 1e9, 1), "frac_hbm": round(byts / t / hbm, 4)})
    del Xb
    # PixArt-alpha's hidden-state shape (8192 x 1152, 18.9 MB): eight distinct tensors in turn, so
    # that inputs and codes together (226 MB) exceed L2 between calls on the same tensor
    Xh = [torch.from_numpy(WL.to_fp16(g.standard_t(5, (8192, 1152)))).to(dev) for _ in range(8)]
    timed16 = graph_timer(torch, reps=16)
    for fmt in range(5):
        qb, wb = cl.act_quant_size(8192, 1152, fmt)
        qs = [torch.empty(qb, dtype=torch.uint8, device=dev) for _ in range(8)]
        ws = torch.empty(max(wb, 256), dtype=torch.uint8, device=dev)
        stq = torch.zeros(1, dtype=torch.int32, device=dev)
        turn = [0]

        def call():
            i = turn[0] % 8
            turn[0] += 1
            cl.act_quant(Xh[i], fmt, qact=qs[i], ws=ws, dev_status=stq)

        t = timed16(call) * 1e-3
        byts = 8192 * 1152 * (3 + (1 / 32 if fmt >= 3 else 0))
        out["big"].append({"fmt": fmt, "M": 8192, "K": 1152, "us": round(t * 1e6, 2), "rotating_tensors": 8,
                           "gbs": round(byts / t / 1e9, 1), "frac_hbm": round(byts / t / hbm, 4)})
    del Xh
    tot = {f: [0.0, 0.0] for f in range(5)}
    for (M, K, N) in WL.UNET_STEP_SHAPES:
        X = torch.from_numpy(WL.to_fp16(g.standard_t(7, (M, K)))).to(dev)
        for fmt in range(5):
            t, byts = one(M, K, fmt, X)
            tot[fmt][0] += t
            tot[fmt][1] += byts
            out["unet_step"].append({"fmt": fmt, "M": M, "K": K, "us": round(t * 1e6, 2),
                                     "gbs": round(byts / t / 1e9, 1)})
    for fmt in range(5):
        t, byts = tot[fmt]
        out["unet_aggregate"].append({"fmt": fmt, "us": round(t * 1e6, 1), "gbs": round(byts / t / 1e9, 1),
                                      "frac_hbm": round(byts / t / hbm, 4)})
    return out


def weight_tables(torch, cl, WL, st, hbm, shape=(4608, 1152)):
    """Selection and pack per palette (W8, W4) on one weight tensor (PixArt-alpha fc1, N x K), and
    the fused selection + pack of the one-class W8 palette.  Pack bytes: 2 B read + b/8 B code write
    per weight + 10 B per channel."""
    N, K = shape
    dev = torch.device("cuda", torch.cuda.current_device())
    W = torch.from_numpy(WL.weight_mix_rows(np.random.default_rng(20266000), N, K)).to(dev)
    timed = graph_timer(torch)
    rows = []
    for name, mask, bits in (("W8", cl.PALETTE_W8, 8), ("W4", cl.PALETTE_W4, 4), ("W4 (DiT set)", W4_PALETTE, 4)):
        fmt = torch.empty(N, dtype=torch.uint8, device=dev)
        t_sel = timed(lambda: cl.select_weight_formats(W, mask, fmt_out=fmt)) * 1e-3
        d = cl.pack_plan(N, K, fmt.cpu().numpy())
        blob, _ = cl.pack_weights(W, fmt, d, dev_status=st)
        t_pack = timed(lambda: cl.pack_weights(W, fmt, d, dev_status=st, blob=blob)) * 1e-3
        pb = 2 * N * K + N * K * bits / 8 + 10 * N
        row = {"palette": name, "N": N, "K": K, "select_us": round(t_sel * 1e6, 2),
               "select_gbs": round(2 * N * K / t_sel / 1e9, 1), "pack_us": round(t_pack * 1e6, 2),
               "pack_gbs": round(pb / t_pack / 1e9, 1), "pack_frac_hbm": round(pb / t_pack / hbm, 4),
               "formats": {int(f): int(c) for f, c in zip(*np.unique(fmt.cpu().numpy(), return_counts=True))}}
        if mask == cl.PALETTE_W8:
            dp = cl.pack_plan_palette(N, K, mask)
            bp = torch.empty(dp.bytes, dtype=torch.uint8, device=dev)
            tf = timed(lambda: cl.select_pack_palette(W, mask, dp, fmt_out=fmt, blob=bp, dev_status=st)) * 1e-3
            row["select_pack_fused_us"] = round(tf * 1e6, 2)
        rows.append(row)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return rows


def workload_variants(torch, cl, st, pk, probe, reps=20):
    """The other workloads' layer shapes, each selected (4-bit palette of its fork), packed,
    quantized and multiplied on the GPU; per shape the GEMM and the quantizer alone (reps
    graph-captured launches between two events) with their roofline fractions (the f16 one, and
    for 8-bit activations the FP8 one: max(flops / peak, bytes / HBM)).  SDXL-UNet W4A8: the 22
    distinct shapes of one step, at a mid bucket (E4M3, dynamic scales); PixArt-alpha W4A8: the
    5 distinct shapes of a block, E5M2 with the DiT path's two per-sample scales; SDXL-Turbo
    weight-only W4A16 rows at batch 1 to 16 (fp16 activations, no quantizer).  Each workload also
    gets its aggregate over its shapes (sum of flops over sum of GEMM times, one launch each)."""
    from paper_2609_33496_gb300 import workloads as WL
    dev = torch.device("cuda", torch.cuda.current_device())
    hbm = pk["hbm_gbs"] * 1e9
    p16 = (probe or {}).get("f16", pk.get("bf16_tflops", 1900.0)) * 1e12
    p8 = (probe or {}).get("f8f6f4", 2 * p16 / 1e12) * 1e12
    palette = (1 << cl.W_INT4_SYM) | (1 << cl.W_INT4_ASYM) | (1 << cl.W_NF4) | (1 << cl.W_E2M1) | \
        (1 << cl.W_MXINT4) | (1 << cl.W_MXFP4)

    def timed(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(reps):
                fn()
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps * 1e-3  # seconds per launch

    turbo = tuple(shp for b in (1, 2, 4, 8, 16) for shp in WL.turbo_batch_shapes(b))
    rows, summary = [], []
    for cfg, name, shapes, af, groups in ((3, "sdxl-unet W4A8", WL.UNET_STEP_SHAPES, cl.A_E4M3, 1),
                                          (4, "pixart-alpha W4A8", WL.PIXART_STEP_SHAPES, cl.A_E5M2, 2),
                                          (5, "sdxl-turbo W4A16", turbo, cl.A_FP16, 1)):
        tot_fl, tot_t, tot_q = 0.0, 0.0, 0.0
        hist = {}
        for i, (M, K, N) in enumerate(shapes):
            X, W, bias = WL.config_layer(cfg, i, M, K, N)
            Xd, Wd, bd = (torch.from_numpy(v).to(dev) for v in (X, W, bias))
            fmt, _ = cl.select_weight_formats(Wd, palette)
            fmt_h = fmt.cpu().numpy()
            for f, c in zip(*np.unique(fmt_h, return_counts=True)):
                hist[int(f)] = hist.get(int(f), 0) + int(c)
            desc = cl.pack_plan(N, K, fmt_h)
            blob, _ = cl.pack_weights(Wd, fmt, desc, dev_status=st)
            ws = torch.empty(cl.linear_workspace_size(M, desc, af), dtype=torch.uint8, device=dev)
            Y = torch.empty((M, N), dtype=torch.float32, device=dev)
            g = groups if M % groups == 0 else 1
            cl.linear_prepare_groups(Xd, desc, af, g, ws, st)
            t = timed(lambda: cl.linear_gemm_ex(Xd, desc, blob, af, g, bd, Y, ws, st))
            fl = 2.0 * M * K * N
            byts = M * K * (2 if af == cl.A_FP16 else 1) + N * K / 2 + 9 * N + 4 * M * N
            row = {"workload": name, "M": M, "K": K, "N": N, "act_fmt": af, "gemm_us": round(t * 1e6, 2),
                   "tflops": round(fl / t / 1e12, 1), "bound": "tensor" if fl / p16 >= byts / hbm else "hbm",
                   "frac_f16_roofline": round(max(fl / p16, byts / hbm) / t, 4)}
            if af != cl.A_FP16:
                row["frac_fp8_roofline"] = round(max(fl / p8, byts / hbm) / t, 4)
                tq = timed(lambda: cl.linear_prepare_groups(Xd, desc, af, g, ws, st))
                tot_q += tq
                row.update({"quant_us": round(tq * 1e6, 2), "quant_gbs": round(4 * M * K / tq / 1e9, 1),
                            "quant_frac_hbm": round(4 * M * K / tq / hbm, 4)})
            rows.append(row)
            tot_fl += fl
            tot_t += t
            del Xd, Wd, bd, blob, ws, Y
        summary.append({"workload": name, "shapes": len(shapes), "gemm_tflops": round(tot_fl / tot_t / 1e12, 1),
                        "gemm_ms": round(tot_t * 1e3, 3), "quant_ms": round(tot_q * 1e3, 3),
                        "weight_formats": dict(sorted(hist.items()))})
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    return {"shapes": rows, "summary": summary}


def dit_grouped(torch, cl, st, steps=20):
    """The DiT path end to end on the 5 GEMMs of a PixArt-alpha block: per linear, input-channel
    energies from the calibration activations of all 10 buckets (GPU), the (g, f) search over
    {32, ..., 288} x {INT4-asym, NF4, E2M1} scored by the input-aware SQNR, the group-wise pack;
    per (layer, bucket) the format the route picks from kappa and SNR on the linear schedule
    (the LUT of Alg. 1); then a 20-step sampler (t_i = 999 - 50 i) in which every step quantizes
    each layer's input with the two samples' own scales (Alg. 3 per sample) in F[l, b(t)] and
    multiplies (fp32 outputs).  The 20 steps are one CUDA graph, timed after a warm replay."""
    from paper_2609_33496_gb300 import workloads as WL
    dev = torch.device("cuda", torch.cuda.current_device())
    snr = cl.snr(cl.SCHEDULE_LINEAR, 1000)
    palette = (1 << cl.W_INT4_ASYM) | (1 << cl.W_NF4) | (1 << cl.W_E2M1)
    gmask = cl.group_mask(cl.GROUP_SIZES)
    cands = cl.group_candidates(palette, gmask)
    layers = []
    for li, (M, K, N) in enumerate(WL.PIXART_STEP_SHAPES):
        W, bias = WL.pixart_layer_weights(li)
        Wd, bd = torch.from_numpy(W).to(dev), torch.from_numpy(bias).to(dev)
        Xs = [torch.from_numpy(WL.pixart_layer_activation(li, b)).to(dev) for b in range(10)]
        energy = torch.zeros(K, dtype=torch.float64, device=dev)
        lut = []
        for b, X in enumerate(Xs):
            cl.act_channel_energy(X, energy=energy)
            sums = cl.act_moments(X).cpu().numpy()
            lut.append(cl.route(cl.kurtosis(sums[:5]), snr[b * 100 + 50], False))
        g, f = cands[cl.candidate_argmin(cl.select_weight_groups(Wd, palette, gmask, energy=energy).cpu().numpy())]
        desc = cl.pack_plan_grouped(N, K, f, g)
        blob, _ = cl.pack_weights(Wd, torch.full((N,), f, dtype=torch.uint8, device=dev), desc, dev_status=st)
        ws = torch.empty(max(cl.linear_workspace_size(M, desc, a) for a in range(6)), dtype=torch.uint8, device=dev)
        Y = torch.empty((M, N), dtype=torch.float32, device=dev)
        layers.append({"Xs": Xs, "desc": desc, "blob": blob, "bias": bd, "ws": ws, "Y": Y, "lut": lut,
                       "g": g, "f": f, "M": M, "K": K, "N": N})
    ts = [999 - 50 * i for i in range(steps)]

    def run():
        for t in ts:
            b = cl.bucket(t)
            for L in layers:
                af = int(L["lut"][b])
                X = L["Xs"][b]
                cl.linear_prepare_groups(X, L["desc"], af, 2, L["ws"], st)
                cl.linear_gemm_ex(X, L["desc"], L["blob"], af, 2, L["bias"], L["Y"], L["ws"], st)

    run()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run()
    g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    g.replay()
    e1.record()
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    ms = e0.elapsed_time(e1)
    flops = steps * sum(2.0 * L["M"] * L["K"] * L["N"] for L in layers)
    used = sorted(set(int(L["lut"][cl.bucket(t)]) for t in ts for L in layers))
    return {"steps": steps, "ms": round(ms, 3), "tflops": round(flops / (ms * 1e-3) / 1e12, 1),
            "weights_g_f": [[L["g"], L["f"]] for L in layers], "lut": [[int(v) for v in L["lut"]] for L in layers],
            "activation_formats_used": used,
            "shapes": [[L["M"], L["K"], L["N"]] for L in layers]}


def tensor_probe(torch, device):
    """Dense tcgen05 throughput this GPU sustains for the GEMM's instruction forms (the probe
    library of the build): kind::f16 (fp16 operands, the W8A8 path) and kind::f8f6f4 (E4M3),
    M = 128, N = 192, on seeded finite operands; and, at the FP8 GEMM's N = 160, the forms that
    GEMM issues: A from tensor memory (TS), with and without UE8M0 block scaling, and the
    block-scaled form with A from shared memory; at N = 192 the TS block-scaled form alone, with
    the GEMM's per-chunk commit + barrier wait + fence after every four MMAs, and the same from
    two issuing threads into two accumulators.  Returns TFLOP/s per form."""
    import ctypes
    from paper_2609_33496_gb300 import build as B
    L = ctypes.CDLL(B.PROBE_LIB)
    L.chameleon_probe_mma.argtypes = [ctypes.c_int] * 4 + [ctypes.c_void_p] * 3
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    cyc = torch.zeros(1, dtype=torch.int64, device=device)
    st = torch.zeros(1, dtype=torch.int32, device=device)
    s = torch.cuda.current_stream()
    out = {}
    for kind, name, K, N in ((0, "f16", 16, 192), (2, "f8f6f4", 32, 192), (3, "f8f6f4_ts_n160", 32, 160),
                             (4, "mxf8f6f4_ts_n160", 32, 160), (5, "mxf8f6f4_ss_n160", 32, 160),
                             (4, "mxf8f6f4_ts_n192", 32, 192), (6, "mxf8f6f4_ts_n192_per_chunk_commit_wait", 32, 192),
                             (7, "mxf8f6f4_ts_n192_per_chunk_commit_wait_two_issuers", 32, 192)):
        iters, best = 4000, 0.0
        for _ in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            rc = L.chameleon_probe_mma(kind, N, sms, iters, ctypes.c_void_p(cyc.data_ptr()),
                                       ctypes.c_void_p(st.data_ptr()), ctypes.c_void_p(s.cuda_stream))
            e1.record(s)
            torch.cuda.synchronize()
            if rc != 0 or int(st.item()) != 0:
                return None
            best = max(best, sms * iters * 4 * 2.0 * 128 * N * K / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        out[name] = round(best, 1)
    return out


# ------------------------------------------------------------------ end to end through host buffers
def pixart_e2e(args, torch, cl, WL, host, lut, device, world, flops_step):
    """The headline step through the public calls with HOST buffers.  Every benchmark step copies
    all 282 layers' weights and biases host->device from pinned memory (then selection and pack),
    and every sampler step copies that step's input tensors host->device and reads the last
    linear's output (block 27 fc2, the step's result) back device->host.  The copies run on their
    own streams beside the compute, as a serving loop would run them:
    * the fp16 weights are read only by selection and pack, so the next step's weights upload
      while this step's sampler runs, one slice behind each sampler step's inputs on the input
      stream (the first timed step's weights were uploaded by the last warm-up step, and the last
      timed step uploads weights for a step that is not run: one 1.2 GB upload per timed step all
      the same); the biases, which the sampler reads, upload at the start of the step;
    * one sampler step's inputs upload while the previous sampler step's linears run (two input
      buffers), and each result is read back on a third stream (two result buffers);
    * each sampler step's 171 `chameleon_linear` calls (quantizer + GEMM per call, as
      `linear_ex` issues them) are captured once in a CUDA graph and replayed, so the host does
      not pace the GPU; selection and pack are issued eagerly every step."""
    import torch.distributed as dist
    Wn, bn, Xn = host
    linears = WL.pixart_model_gemms()
    n = len(linears)
    keys = sorted(WL.PIXART_INPUTS)
    ts = WL.PIXART_SAMPLER_T[:args.sampler_steps]
    buckets = [cl.bucket(t) for t in ts]
    Wh = [torch.from_numpy(np.concatenate([Wn[i] for i in ix])).pin_memory() for (_, M, K, N, _, ix) in linears]
    bh = [torch.from_numpy(np.concatenate([bn[i] for i in ix])).pin_memory() for (_, M, K, N, _, ix) in linears]
    Xh = {kb: torch.from_numpy(x).pin_memory() for kb, x in Xn.items() if kb[1] in set(buckets)}
    Wd = [torch.empty_like(w, device=device) for w in Wh]
    bd = [torch.empty_like(b, device=device) for b in bh]
    # zero-filled: the pass before the graphs are captured runs on them (finite values)
    Xd = [{k: torch.zeros(WL.PIXART_INPUTS[k], dtype=torch.float16, device=device) for k in keys} for _ in range(2)]
    last = linears[-1]
    Yd_last = [torch.empty((last[1], last[3]), dtype=torch.float32, device=device) for _ in range(2)]
    Yh = [torch.empty((last[1], last[3]), dtype=torch.float32).pin_memory() for _ in range(2)]
    st = torch.zeros(1, dtype=torch.int32, device=device)
    offs = np.cumsum([0] + [N for (_, M, K, N, _, _) in linears])
    fmt_all = torch.empty(int(offs[-1]), dtype=torch.uint8, device=device)
    fmt_host = torch.empty(int(offs[-1]), dtype=torch.uint8).pin_memory()
    compute = torch.cuda.current_stream()
    copy = torch.cuda.Stream(device)       # input and bias uploads
    wcopy = torch.cuda.Stream(device)      # weight uploads (the inputs are not queued behind them)
    readback = torch.cuda.Stream(device)   # result read-backs (not queued behind the next uploads)
    for i in range(n):
        Wd[i].copy_(Wh[i])
        bd[i].copy_(bh[i])
    for i in range(n):
        cl.select_weight_formats(Wd[i], W4_PALETTE, fmt_out=fmt_all[offs[i]:offs[i + 1]])
    f_ref = fmt_all.cpu().numpy()
    descs = [cl.pack_plan(N, K, f_ref[offs[i]:offs[i + 1]]) for i, (_, M, K, N, _, _) in enumerate(linears)]
    blobs = [torch.empty(d.bytes, dtype=torch.uint8, device=device) for d in descs]
    for i in range(n):
        cl.pack_weights(Wd[i], fmt_all[offs[i]:offs[i + 1]], descs[i], dev_status=st, blob=blobs[i])
    acts = sorted(set(lut.values()))
    ws = torch.empty(max(cl.linear_workspace_size(M, descs[i], a) for i, (_, M, K, N, _, _) in enumerate(linears)
                         for a in acts), dtype=torch.uint8, device=device)
    kind = [names[0].split(".", 1)[1] if names[0].startswith("block") else names[0] for (names, *_r) in linears]
    Ys = {}
    for k, (names, M, K, N, _, _) in zip(kind[:-1], linears[:-1]):
        if k not in Ys:
            Ys[k] = torch.empty((M, N), dtype=torch.float32, device=device)
    Y = [Ys[k] for k in kind[:-1]]              # the last linear writes Yd_last (two buffers)
    x_ready = [torch.cuda.Event() for _ in range(2)]
    x_free = [torch.cuda.Event() for _ in range(2)]
    y_ready = [torch.cuda.Event() for _ in range(2)]
    y_read = [torch.cuda.Event() for _ in range(2)]
    w_ready, b_ready, packed = torch.cuda.Event(), torch.cuda.Event(), torch.cuda.Event()
    h2d = sum(w.numel() * 2 + b.numel() * 4 for w, b in zip(Wh, bh)) + \
        sum(Xh[(k, b)].numel() * 2 for b in buckets for k in keys)
    d2h = len(buckets) * Yh[0].numel() * 4

    def sampler_step(s, b):
        buf = s % 2
        for i, (names, M, K, N, key, _) in enumerate(linears):
            yi = Yd_last[buf] if i == n - 1 else Y[i]
            cl.linear_ex(Xd[buf][key], descs[i], blobs[i], lut[(key, b)], 2, bias=bd[i], Y=yi, ws=ws,
                         dev_status=st)

    for s, b in enumerate(buckets):              # eager once, then captured
        sampler_step(s, b)
    torch.cuda.synchronize()
    if int(st.item()) != 0:
        raise RuntimeError("device status %d before capture" % int(st.item()))
    graphs = []
    for s, b in enumerate(buckets):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            sampler_step(s, b)
        graphs.append(g)
    torch.cuda.synchronize()
    st.zero_()

    wslices = np.array_split(np.arange(n), len(buckets))

    def upload_weights():
        with torch.cuda.stream(wcopy):
            wcopy.wait_event(packed)             # selection and pack have read the weights
            for i in range(n):
                Wd[i].copy_(Wh[i], non_blocking=True)
            w_ready.record(wcopy)

    def step():
        with torch.cuda.stream(copy):
            copy.wait_stream(compute)            # the previous sampler no longer reads the biases
            for i in range(n):
                bd[i].copy_(bh[i], non_blocking=True)
            b_ready.record(copy)
        compute.wait_event(w_ready)              # this step's weights (uploaded during the last one)
        for i in range(n):
            cl.select_weight_formats(Wd[i], W4_PALETTE, fmt_out=fmt_all[offs[i]:offs[i + 1]])
        fmt_host.copy_(fmt_all, non_blocking=True)
        compute.synchronize()
        if not np.array_equal(fmt_host.numpy(), f_ref):
            raise RuntimeError("the selected formats changed between steps")
        for i in range(n):
            cl.pack_weights(Wd[i], fmt_all[offs[i]:offs[i + 1]], descs[i], dev_status=st, blob=blobs[i])
        packed.record(compute)
        compute.wait_event(b_ready)
        for s, b in enumerate(buckets):
            buf = s % 2
            with torch.cuda.stream(copy):
                copy.wait_event(x_free[buf])
                for k in keys:
                    Xd[buf][k].copy_(Xh[(k, b)], non_blocking=True)
                x_ready[buf].record(copy)
                # the next step's weights, one slice behind each sampler step's inputs on the same
                # stream: the inputs, which the next sampler step waits for, go first on the link
                if s == 0:
                    copy.wait_event(packed)      # selection and pack have read the weights
                for i in wslices[s]:
                    Wd[i].copy_(Wh[i], non_blocking=True)
                if s == len(buckets) - 1:
                    w_ready.record(copy)
            compute.wait_event(x_ready[buf])
            compute.wait_event(y_read[buf])      # the result buffer's previous read-back is done
            graphs[s].replay()
            x_free[buf].record(compute)
            y_ready[buf].record(compute)
            with torch.cuda.stream(readback):    # the step's result, read back beside the next step
                readback.wait_event(y_ready[buf])
                Yh[buf].copy_(Yd_last[buf], non_blocking=True)
                y_read[buf].record(readback)
        compute.wait_stream(readback)            # every read-back of the step has landed

    for e in x_free + y_read + [packed]:
        e.record(compute)
    upload_weights()
    for _ in range(max(1, args.warmup - 1)):
        step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(compute)
    for _ in range(args.steps):
        step()
    compute.wait_stream(copy)                    # the uploads issued in the timed steps have landed
    t1.record(compute)
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    if world > 1:
        ms = max_over_ranks(ms, device)
    if int(st.item()) != 0:
        raise RuntimeError("device status %d after the e2e steps" % int(st.item()))
    # the last read-back holds the final sampler step's result of block 27 fc2
    buf = (len(buckets) - 1) % 2
    if not np.isfinite(Yh[buf].numpy()).all():
        raise RuntimeError("non-finite values in the step's result")
    # host->device bandwidth alone, after the timed steps: the step's weight uploads twice over,
    # nothing else running; h2d / that rate is the copy time a step cannot go below
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wbytes = sum(w.numel() * 2 for w in Wh)
    with torch.cuda.stream(wcopy):
        e0.record(wcopy)
        for _ in range(2):
            for i in range(n):
                Wd[i].copy_(Wh[i], non_blocking=True)
        e1.record(wcopy)
    torch.cuda.synchronize()
    h2d_gbs = 2 * wbytes / (e0.elapsed_time(e1) * 1e-3) / 1e9
    return {"value": round(job_tflops(flops_step, args.steps, world, ms), 3), "unit": "TFLOP/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "ms_per_step": round(ms / args.steps, 3),
            "calls": "chameleon_select_weight_formats, chameleon_pack_plan, chameleon_pack_weights, "
                     "chameleon_linear_prepare_groups + chameleon_linear_gemm_ex (each sampler step's calls "
                     "captured once in a CUDA graph)",
            "pipelining": "next step's weights upload during this step's sampler; inputs double-buffered; "
                          "read-backs on a third stream",
            "h2d_gbs_alone": round(h2d_gbs, 2),
            "h2d_ms_per_step_at_that_rate": round(h2d / (h2d_gbs * 1e9) * 1e3, 1)}


# ------------------------------------------------------------------ the oracle as CPU baseline
def oracle_sample(which=("block0.self.q", "block0.cross.k", "caption.fc1"), buckets=(0, 9)):
    """The oracle on a bounded sample of the headline workload: for each linear of the sample,
    per-channel selection over the 4-bit palette and the pack (the selected formats' codes and
    scales, decoded to their exact values) once, as the GPU step does; then at each bucket the
    quantizer per sample (Alg. 3) in the format the route picks and the fp64 GEMM over all rows.
    Each stage timed.  Returns (flops, seconds, description, seconds per stage)."""
    from oracle import formats as F
    from oracle import gemm as G
    from oracle import schedule as S
    from oracle import select as SEL
    from paper_2609_33496_gb300 import workloads as WL
    snr = S.snr(S.betas_linear())
    linears = WL.pixart_model_linears()
    idx = [next(i for i, L in enumerate(linears) if L[0] == w) for w in which]
    flops, stages = 0.0, {"select": 0.0, "pack": 0.0, "act_quant": 0.0, "gemm": 0.0}
    for i in idx:
        name, M, K, N, key = linears[i]
        W, bias = WL.pixart_model_weights(i)
        t0 = time.perf_counter()
        fmt, _, _ = SEL.select_formats(W, W4_PALETTE)
        t1 = time.perf_counter()
        w = SEL.dequant_selected(W, fmt)
        t2 = time.perf_counter()
        stages["select"] += t1 - t0
        stages["pack"] += t2 - t1
        for b in buckets:
            X = WL.pixart_model_input(key, b)
            f = S.route(S.kurtosis(X), snr[int(S.bucket_midpoint(b))])  # calibration: outside the timed path
            t2 = time.perf_counter()
            a = F.act_dequant_per_sample(F.act_quant_per_sample(X, f, 2))
            t3 = time.perf_counter()
            G.linear_output(a, w, bias)
            t4 = time.perf_counter()
            stages["act_quant"] += t3 - t2
            stages["gemm"] += t4 - t3
            flops += layer_flops(M, K, N)
    desc = ("oracle select (4-bit palette) + pack of %s, then per-sample act-quant + fp64 GEMM at buckets %s"
            % (list(which), list(buckets)))
    return flops, sum(stages.values()), desc, stages


def cpu_baseline(cores):
    """The oracle sample timed twice, in child processes: on one core (one BLAS thread) and on all
    of the host's cores (BLAS threads = cores; selection, pack and quantizer are single-threaded
    numpy either way)."""
    out = {}
    for threads in (1, cores):
        env = dict(os.environ, OPENBLAS_NUM_THREADS=str(threads), OMP_NUM_THREADS=str(threads),
                   MKL_NUM_THREADS=str(threads))
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample"], env=env,
                           capture_output=True, text=True, timeout=600)
        out[threads] = json.loads(r.stdout.strip().splitlines()[-1])
    allc, one = out[cores], out[1]
    return {"value": allc["value"], "unit": "TFLOP/s", "cores": cores, "kind": "oracle", "sample": allc["sample"],
            "seconds": allc["seconds"], "stage_seconds": allc["stage_seconds"],
            "single_core": {"value": one["value"], "seconds": one["seconds"], "stage_seconds": one["stage_seconds"]},
            "host_cores": os.cpu_count()}


def oracle_sample_main():
    flops, t, desc, stages = oracle_sample()
    print(json.dumps({"value": round(flops / t / 1e12, 6), "seconds": round(t, 2), "sample": desc,
                      "stage_seconds": {k: round(v, 3) for k, v in stages.items()}}))
    return 0


def reference_arm(args, world):
    """The oracle as the reference arm (the paper ships no code): each step one bucket of the
    sample, on this process's one BLAS thread."""
    for _ in range(args.warmup):
        oracle_sample(buckets=(9,))
    flops, t, desc = 0.0, 0.0, ""
    for _ in range(args.steps):
        f, s, desc, _ = oracle_sample(buckets=(9,))
        flops += f
        t += s
    value = flops / t / 1e12
    return {"metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(1e3 * t / args.steps, 2), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": WORKLOAD, "sample": desc},
            "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# ------------------------------------------------------------------ single kernel cases for profilers
PROFILE_CASES = {
    "gemm-pixart-qkv": "the stacked q/k/v GEMM of a PixArt-alpha block (8192 x 1152 x 3456), the 4-bit palette's "
                       "per-channel selection, E4M3 activations with two per-sample scales: 3 GEMM launches",
    "gemm-pixart-fc1": "PixArt-alpha fc1 (8192 x 1152 x 4608), as above: 3 GEMM launches",
    "gemm-sdxl-geglu": "SDXL GEGLU-in (2048 x 1280 x 10240), W8 palette, E4M3: 3 GEMM launches (fp16 kernel)",
    "quant-pixart-fc2": "the dynamic per-sample quantizer (range + encode) of PixArt-alpha fc2's input (8192 x 4608, "
                        "E4M3, codes + fp16 operand for a layer with NF4 tiles): 3 calls",
    "quant-pixart-hidden": "the dynamic per-sample quantizer of a PixArt-alpha hidden-state input (8192 x 1152, E4M3, "
                           "codes + fp16 operand): one cooperative launch, 3 calls",
    "pack-w4": "selection and pack of PixArt-alpha fc1's weights (4608 x 1152) over the 4-bit palette: 3 pack launches",
    "gemm-small-m16": "16 tokens x 1280 x 1280 (the small-M weight-streaming kernel), 4-bit palette, E4M3 with two "
                      "per-sample scales: 3 GEMM launches",
}


def profile_case(name):
    """Run one named case a few times (after one warm call) for a profiler; prints 'ok'."""
    import torch
    import paper_2609_33496_gb300 as P
    from paper_2609_33496_gb300 import build as B
    from paper_2609_33496_gb300 import workloads as WL
    B.build()
    cl = P.chameleon
    dev = torch.device("cuda", 0)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    g = np.random.default_rng(20267000)
    shapes = {"gemm-pixart-qkv": (8192, 1152, 3456, W4_PALETTE), "gemm-pixart-fc1": (8192, 1152, 4608, W4_PALETTE),
              "gemm-sdxl-geglu": (2048, 1280, 10240, cl.PALETTE_W8), "quant-pixart-fc2": (8192, 4608, 1152, W4_PALETTE),
              "quant-pixart-hidden": (8192, 1152, 1152, W4_PALETTE),
              "pack-w4": (8192, 1152, 4608, W4_PALETTE), "gemm-small-m16": (16, 1280, 1280, W4_PALETTE)}
    M, K, N, pal = shapes[name]
    X = torch.from_numpy(WL.to_fp16(g.standard_t(7, (M, K)))).to(dev)
    W = torch.from_numpy(WL.weight_mix_rows(g, N, K)).to(dev)
    fmt, _ = cl.select_weight_formats(W, pal)
    d = cl.pack_plan(N, K, fmt.cpu().numpy())
    blob, _ = cl.pack_weights(W, fmt, d, dev_status=st)
    ws = torch.empty(cl.linear_workspace_size(M, d, cl.A_E4M3), dtype=torch.uint8, device=dev)
    Y = torch.empty((M, N), dtype=torch.float32, device=dev)
    groups = 1 if name == "gemm-sdxl-geglu" else 2
    cl.linear_prepare_groups(X, d, cl.A_E4M3, groups, ws, st)
    for _ in range(4):
        if name.startswith("gemm"):
            cl.linear_gemm_ex(X, d, blob, cl.A_E4M3, groups, None, Y, ws, st)
        elif name.startswith("quant"):
            cl.linear_prepare_groups(X, d, cl.A_E4M3, groups, ws, st)
        else:
            cl.pack_weights(W, fmt, d, dev_status=st, blob=blob)
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    print("ok", name)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-variants", action="store_true", help="skip the sub-objects (config 2, per-variant tables)")
    ap.add_argument("--sampler-steps", type=int, default=20, help="sampler steps per benchmark step (smaller cases)")
    ap.add_argument("--oracle-sample", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--case", choices=sorted(PROFILE_CASES), help="run one kernel case for a profiler and exit")
    args = ap.parse_args()
    if args.oracle_sample:
        return oracle_sample_main()
    if args.case:
        return profile_case(args.case)
    args.warmup = max(args.warmup, 3)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(reference_arm(args, world)), flush=True)
        return 0

    cores = os.cpu_count() or 1
    host = pixart_host_inputs(max(1, min(16, cores // max(1, world))))   # before this process touches the GPU

    import torch
    import torch.distributed as dist
    import paper_2609_33496_gb300 as P
    from paper_2609_33496_gb300 import build as B
    from paper_2609_33496_gb300 import workloads as WL

    B.build()
    cl = P.chameleon
    cl.lib()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)
    st = torch.zeros(1, dtype=torch.int32, device=device)
    pk, pk_kind = peaks()
    h = pixart_headline(args, torch, cl, WL, host, device, world, st)
    K_ = args.steps
    probe = tensor_probe(torch, device)

    # roofline of the GEMM class: every linear is tensor-bound; class-0 tiles run FP8 MMAs (peak =
    # the measured bf16 rate x the nominal FP8 / bf16 ratio), NF4 tiles fp16 MMAs (the bf16 rate)
    gemm_ms = h["classes_ms"]["g"]
    achieved = h["flops_step"] / (gemm_ms * 1e-3) / 1e12
    p16s, p16b = pk.get("bf16_tflops_sustained", pk["bf16_tflops"]), pk["bf16_tflops"]
    t_roof_s = h["fl8"] / (FP8_OVER_BF16 * p16s) + h["fl16"] / p16s
    t_roof_b = h["fl8"] / (FP8_OVER_BF16 * p16b) + h["fl16"] / p16b
    peak_eff_s = h["flops_step"] / t_roof_s   # TFLOP/s: the peaks above are in TFLOP/s
    peak_eff_b = h["flops_step"] / t_roof_b
    hbm = pk["hbm_gbs"] * 1e9
    qgbs = h["qbytes"] / (h["classes_ms"]["q"] * 1e-3) / 1e9
    lut_by_bucket = {}
    for (key, b), f in sorted(h["lut"].items()):
        lut_by_bucket.setdefault(b, {})[key] = f
    result = {
        "metric": METRIC, "value": round(h["value_tflops"], 3), "unit": "TFLOP/s", "n_gpus": world, "steps": K_,
        "warmup": args.warmup, "ms_per_step": round(h["elapsed_ms"] / K_, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "fp8 (e4m3 x e4m3/e5m2 MMA, fp32 accumulate; fp16 on NF4 tiles)",
        "data": "synthetic (seeded random-init weights, Student-t activations)",
        "config": {"workload": WORKLOAD if args.sampler_steps == 20 else WORKLOAD + " (%d sampler steps)" % args.sampler_steps,
                   "model": "PixArt-alpha-architecture DiT", "linears": h["n_linears"], "gemms": len(h["linears"]),
                   "stacked": "q/k/v and cross k/v of each block read the same input: one quantizer pass and one "
                              "GEMM with their weights stacked along N (per-channel formats and outputs unchanged)",
                   "sampler_steps": len(h["buckets"]), "global_batch": 2 * world, "tokens": [8192, 240],
                   "weight_palette": "W4 {INT4-asym, NF4, E2M1, MXINT4, MXFP4}, per-channel argmin",
                   "weight_formats": h["weight_formats"],
                   "lut": {str(b): v for b, v in lut_by_bucket.items()},
                   "activation_formats_used": h["acts"],
                   "step": "selection + pack of the 282 layers, then 20 sampler steps x 171 GEMMs (per-sample "
                           "dynamic quantizer + GEMM, one CUDA graph)",
                   "l2": "inputs larger than L2 (1.7 GB of activations, 0.3 GB of packed weights)",
                   "parallelism": "replicas" if world > 1 else "single-gpu"},
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": round(peak_eff_s, 1), "unit": "TFLOP/s",
                     "frac": round(achieved / peak_eff_s, 4), **traffic_fields(),
                     "kernel": "k_gemm_ts_f8 (tcgen05 kind::mxf8f6f4 on class-0 tiles, kind::f16 on NF4 tiles)",
                     "peak_source": ("%s bf16_tflops_sustained x %.0f for the FP8 share of the flops, x 1 for the "
                                     "fp16 share (the GEMM class runs ~%.0f ms per replay, back to back)"
                                     % (pk_kind, FP8_OVER_BF16, gemm_ms)),
                     "fp8_flop_share": round(h["fl8"] / h["flops_step"], 4),
                     "frac_burst": round(achieved / peak_eff_b, 4), "peak_burst": round(peak_eff_b, 1),
                     "gemm_ms_per_step": round(gemm_ms, 3), "probe_tflops": probe,
                     "timing": "value: selection + pack (two CUDA-graph replays, the formats checked on the host) and one CUDA-graph replay of the sampler per step; "
                               "GEMM class: the sampler's GEMM launches alone, graph-replayed once per timed step"},
        "act_quant": {"achieved_gbs": round(qgbs, 1), "peak_gbs": pk["hbm_gbs"], "frac": round(qgbs * 1e9 / hbm, 4),
                      "ms_per_step": round(h["classes_ms"]["q"], 3),
                      "bytes": "algorithmic: 2 B read + 1 B code per element (+1/32 B MX); the path also writes the "
                               "exact fp16 operand for NF4 tiles (not counted)"},
        "weights_select_pack_ms_per_step": round(h["classes_ms"]["w"], 3),
        "gpu_launches": h["launches"] * K_,
        "clocks": h["clocks"],
    }
    if not args.no_variants:
        p16 = (probe or {}).get("f16", p16b) * 1e12
        p8 = (probe or {}).get("f8f6f4", FP8_OVER_BF16 * p16b) * 1e12
        result["sdxl_w8a8"] = sdxl_step(args, torch, cl, WL, device, st, pk)
        result["variants"] = {"gemm": gemm_matrix(torch, cl, WL, st, p16, p8, hbm),
                              "quant": quant_tables(torch, cl, WL, hbm),
                              "weights": weight_tables(torch, cl, WL, st, hbm),
                              "workloads": workload_variants(torch, cl, st, pk, probe),
                              "dit_grouped": dit_grouped(torch, cl, st)}
    if not args.no_e2e:
        result["e2e"] = pixart_e2e(args, torch, cl, WL, host, h["lut"], device, world, h["flops_step"])
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(cores)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

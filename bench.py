#!/usr/bin/env python
"""Benchmark of the Chameleon format-adaptive quantized linear path on GB300.

Workload: the SDXL-UNet attention/FFN projections at batch 2 with classifier-free guidance, W8A8
(q/k/v/out 8192x640x640 x4, 2048x1280x1280 x4, GEGLU-in 2048x1280->10240, FF-out 2048x5120->1280),
seeded synthetic activations over the 10 timestep buckets.  One step is one pass of the whole hot
path: per-channel weight-format selection and pack of all 10 layers, then for every bucket and
layer the activation quantizer in the format the (layer, bucket) LUT picks and the tcgen05 GEMM.

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

os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")   # the oracle's timed leg runs on one core
os.environ.setdefault("OMP_NUM_THREADS", "1")

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "mixed-format linear TFLOP/s & % tensor peak; act-quant HBM GB/s"
WORKLOAD = "SDXL-UNet attention/FFN projections, W8A8, batch 2 (CFG), 10 timestep buckets"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_BYTES = 126 * 2 ** 20
# dram__bytes_read.sum + dram__bytes_write.sum of one launch of the dominant kernel, from an ncu
# capture of the GEGLU-in projection (M 2048, K 1280, N 10240; profiles/gemm_ts_f16_sdxl_geglu_in.md).
# Set to None whenever the kernel changes until it is captured again.
GEMM_TRAFFIC_PER_LAUNCH = {"bytes": 43.79e6, "launch": "2048x1280x10240 (GEGLU-in)",
                           "algorithmic_bytes": 99.8e6}


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


# ------------------------------------------------------------------ workload
def layer_flops(M, K, N):
    return 2.0 * M * K * N


def host_inputs(WL, layer_ids, buckets):
    """Weights, biases and the activations of every (layer, bucket), generated once on the host."""
    Wn, bn, Xn = [], [], []
    for li in layer_ids:
        w, b = WL.sdxl_layer_weights(li)
        Wn.append(w)
        bn.append(b)
        Xn.append([WL.sdxl_layer_activation(li, bk) for bk in buckets])
    return Wn, bn, Xn


def build_inputs(torch, host, device):
    Wn, bn, Xn = host
    W = [torch.from_numpy(w).to(device) for w in Wn]
    bias = [torch.from_numpy(b).to(device) for b in bn]
    X = [[torch.from_numpy(x).to(device) for x in xs] for xs in Xn]
    return W, bias, X


def calibrate_lut(torch, cl, X, buckets):
    """Alg. 1 on the synthetic activations (the calibration set is the step's own activations):
    power sums and range on the GPU, kappa, SNR at the bucket midpoint (scaled-linear schedule),
    Route -> F[l, b], and the static ScaleZP(F[l, b], lo[l, b], hi[l, b]) that the UNet path
    quantizes with (Alg. 2; None for the MX formats, which carry block exponents instead)."""
    snr = cl.snr(cl.SCHEDULE_SCALED_LINEAR, 1000)
    lut = np.zeros((len(X), len(buckets)), dtype=np.int64)
    kappa = np.zeros((len(X), len(buckets)))
    qp = [[None] * len(buckets) for _ in X]
    sse = np.zeros((len(X), len(buckets), 5))
    for li, xs in enumerate(X):
        for j, x in enumerate(xs):
            sums = cl.act_moments(x).cpu().numpy()
            kappa[li, j] = cl.kurtosis(sums[:5])
            lut[li, j] = cl.route(kappa[li, j], snr[buckets[j] * 100 + 50], False)
            if lut[li, j] <= 2:
                qp[li][j] = cl.scale_zp(int(lut[li, j]), float(sums[5]), float(sums[6]))
            sse[li, j] = cl.act_format_sse(x)[0].cpu().numpy()   # Eq. format-argmin, for comparison
    return lut, kappa, qp, sse


def route_vs_argmin(cl, lut, sse):
    """How the kappa / SNR route (Sec. 3.3) compares with the exhaustive argmin of Eq.
    format-argmin on the same calibration tensors."""
    best = np.array([[cl.act_format_argmin(sse[i, j]) for j in range(sse.shape[1])] for i in range(sse.shape[0])])
    picked = np.take_along_axis(sse, lut[..., None], axis=2)[..., 0]
    opt = np.take_along_axis(sse, best[..., None], axis=2)[..., 0]
    ratio = picked / np.maximum(opt, 1e-300)
    # the same over the per-tensor formats (0..2), the only ones the route picks off the shortcut layers
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
            "per_tensor_argmin_formats": {int(f): int(c) for f, c in zip(*np.unique(best3, return_counts=True))},
            "argmin_formats": {int(f): int(c) for f, c in zip(*np.unique(best, return_counts=True))},
            "route_formats": {int(f): int(c) for f, c in zip(*np.unique(lut, return_counts=True))}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-variants", action="store_true", help="skip the per-variant matrix")
    ap.add_argument("--dynamic-scales", action="store_true",
                    help="quantize with each tensor's own range (Alg. 3, the DiT path) instead of the "
                         "calibrated static scales of the UNet path (Alg. 2)")
    ap.add_argument("--layers", default="all", help="comma-separated layer indices (smaller cases for profiling)")
    ap.add_argument("--buckets", default="all", help="comma-separated timestep buckets")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(reference_arm(args, world)), flush=True)
        return 0

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

    layer_ids = list(range(len(WL.SDXL_PROJ_LAYERS))) if args.layers == "all" else [
        int(v) for v in args.layers.split(",")]
    buckets = list(range(10)) if args.buckets == "all" else [int(v) for v in args.buckets.split(",")]
    layers = [WL.SDXL_PROJ_LAYERS[i] for i in layer_ids]
    nb = len(buckets)
    host = host_inputs(WL, layer_ids, buckets)
    W, bias, X = build_inputs(torch, host, device)
    lut, kappa, qp, cal_sse = calibrate_lut(torch, cl, X, buckets)
    st = torch.zeros(1, dtype=torch.int32, device=device)
    stream = torch.cuda.current_stream()

    # buffers reused every step (the packed weights are re-packed in place every step)
    Y = [torch.empty((M, N), dtype=torch.float32, device=device) for (_, M, K, N) in layers]
    ws = [torch.empty(max(cl.linear_workspace_size(M, cl.pack_plan(N, K, np.zeros(N, np.uint8)), f)
                          for f in range(6)), dtype=torch.uint8, device=device) for (_, M, K, N) in layers]
    blobs, descs = [None] * len(layers), [None] * len(layers)
    fmt_off = np.cumsum([0] + [N for (_, M, K, N) in layers])
    fmt_all = torch.empty(int(fmt_off[-1]), dtype=torch.uint8, device=device)

    # the W8 palette's formats share one MMA class, so the packed layout follows from N, K and
    # the palette: selection and pack need no host round trip and run inside the step's graph
    for li, (_, M, K, N) in enumerate(layers):
        descs[li] = cl.pack_plan_palette(N, K, cl.PALETTE_W8)
        blobs[li] = torch.empty(descs[li].bytes, dtype=torch.uint8, device=device)

    def select_pack():
        """a5 + a6 for every layer in one launch each: GPU selection into the layer's slice of one
        format buffer and, from the same warp, the pack into the layer's blob."""
        for li in range(len(layers)):
            f = fmt_all[fmt_off[li]:fmt_off[li + 1]]
            cl.select_pack_palette(W[li], cl.PALETTE_W8, descs[li], fmt_out=f, blob=blobs[li], dev_status=st)

    flops_step = nb * sum(layer_flops(M, K, N) for (_, M, K, N) in layers)
    quant_bytes_step = 0.0

    def run_step(parts="wqg"):
        """a5 + a6 for every layer ("w"), then a2-a4 + a7 for every (bucket, layer): act-quant in
        F[l, b] with the calibrated static (S, Z)[l, b] of the UNet path ("q") and the GEMM ("g")."""
        if "w" in parts:
            select_pack()
        for bk in range(nb):
            for li, (_, M, K, N) in enumerate(layers):
                f = int(lut[li, bk])
                if "q" in parts:
                    if args.dynamic_scales:
                        cl.linear_prepare(X[li][bk], descs[li], f, ws[li], st)
                    else:
                        cl.linear_prepare_static(X[li][bk], descs[li], f, qp[li][bk], ws[li], st)
                if "g" in parts:
                    cl.linear_gemm(X[li][bk], descs[li], blobs[li], f, bias[li], Y[li], ws[li], st)

    # warm-up (eager), then capture one whole step in a CUDA graph (no event nodes inside: each
    # costs about 5 us of serialisation), plus graphs holding only the selection + pack, only the
    # quantizer and only the GEMM launches of the step, which time those kernel classes
    for _ in range(args.warmup):
        run_step()
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    graphs = {}
    try:
        for key in ("wqg", "w", "q", "g"):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                run_step(key)
            graphs[key] = g
        for _ in range(args.warmup):
            graphs["wqg"].replay()
        torch.cuda.synchronize()
    except RuntimeError as exc:  # a launch that cannot be captured: time eager launches
        print("bench: CUDA-graph capture failed (%s); timing eager launches" % exc, file=sys.stderr)
        graphs = {}
        torch.cuda.synchronize()

    def replay(key):
        if key in graphs:
            graphs[key].replay()
        else:
            run_step(key)

    # kernel launches per step: one fused select + pack per layer (one MMA class: slot = channel);
    # per linear 1 quantizer kernel (static scales or MX; 2 with dynamic per-tensor scales) + 1 GEMM
    launches = len(layers) + sum(
        (2 if args.dynamic_scales and lut[li, bk] <= 2 else 1) + 1 for li in range(len(layers)) for bk in range(nb))
    # the quantizer's algorithmic bytes: X read, the exact fp16 operand written (MX formats fold
    # the block exponent into the operand, so no E8M0 bytes are written on this path)
    for li, (_, M, K, N) in enumerate(layers):
        quant_bytes_step += nb * (M * K * 2 + M * K * 2)
    # ---------------------------------------------------------------- timed region (device)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for k in range(args.steps):
            replay("wqg")
        t1.record(stream)
        torch.cuda.synchronize()
        # kernel classes, each alone: the step's 100 quantizer (or GEMM) launches back to back,
        # replayed as many times as the timed steps, two events around them
        class_ms = {}
        for key in ("g", "q", "w"):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for k in range(args.steps):
                replay(key)
            e1.record(stream)
            torch.cuda.synchronize()
            class_ms[key] = e0.elapsed_time(e1)
    gemm_ms, quant_ms, weights_ms = class_ms["g"], class_ms["q"], class_ms["w"]
    n_linear = nb * len(layers)
    if world > 1:
        dist.barrier()
    elapsed_ms = t0.elapsed_time(t1)
    if world > 1:
        elapsed_ms = max_over_ranks(elapsed_ms, device)
    assert int(st.item()) == 0, "device status %d" % int(st.item())

    K_ = args.steps
    value = job_tflops(flops_step, K_, world, elapsed_ms)
    pk, pk_kind = peaks()
    peak_tensor = pk.get("bf16_tflops_sustained", pk.get("bf16_tflops"))
    gemm_tflops = flops_step * K_ / (gemm_ms * 1e-3) / 1e12
    quant_gbs = quant_bytes_step * K_ / (quant_ms * 1e-3) / 1e9
    # roofline time of every GEMM launch: max(flops / tensor peak, algorithmic bytes / HBM peak)
    t_roof = 0.0
    for li, (_, M, K, N) in enumerate(layers):
        b = M * K + N * K + 5 * N + 4 * N + 4 * M * N
        t_roof += nb * max(layer_flops(M, K, N) / (peak_tensor * 1e12), b / (pk["hbm_gbs"] * 1e9))
    clocks = clk.summary()
    probe = tensor_probe(torch, device)
    variants = None if args.no_variants else variant_matrix(torch, cl, W, bias, X, layers, lut, qp, st, pk, probe)
    if variants is not None:
        variants["workloads"] = workload_variants(torch, cl, st, pk, probe)
        variants["dit_sampler"] = dit_sampler(torch, cl, st)

    result = {
        "metric": METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": world, "steps": K_,
        "warmup": args.warmup, "ms_per_step": round(elapsed_ms / K_, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": WORKLOAD if (args.layers, args.buckets) == ("all", "all") else
                   WORKLOAD + " (subset: layers %s, buckets %s)" % (layer_ids, buckets),
                   "layers": len(layers), "buckets": nb, "global_batch": 2 * world,
                   "tokens": [M for (_, M, _, _) in layers], "weight_palette": "W8 {INT8-sym, INT8-asym, MXINT8}",
                   "activation_formats_used": sorted(set(int(v) for v in lut.ravel())),
                   "lut": [[int(v) for v in row] for row in lut],   # F[layer][bucket] from Alg. 1's route
                   "step": "fused select+pack of 10 layers, then 10 buckets x 10 layers of act-quant (%s) + GEMM, one "
                           "CUDA graph" % ("dynamic per-tensor scales, Alg. 3" if args.dynamic_scales else
                                           "static calibrated per-(layer, bucket) scales, Alg. 2"),
                   "l2": "inputs larger than L2 (%.0f MB of activations per step)" %
                         (sum(x.numel() * 2 for xs in X for x in xs) / 1e6),
                   "parallelism": "replicas" if world > 1 else "single-gpu"},
        "roofline": {"bound": "tensor", "achieved": round(gemm_tflops, 2), "peak": peak_tensor,
                     "unit": "TFLOP/s", "frac": round(gemm_tflops / peak_tensor, 4),
                     **traffic_fields(),
                     "kernel": "k_gemm_ts_f16 (tcgen05 kind::f16, weights decoded into TMEM)",
                     "peak_source": "%s bf16_tflops_sustained (fp16 MMA rate = bf16 rate)" % pk_kind,
                     "roofline_time_frac": round(t_roof * K_ / (gemm_ms * 1e-3), 4),
                     "gemm_ms_per_step": round(gemm_ms / K_, 4),
                     "gemm_launch_ms_mean": round(gemm_ms / (args.steps * n_linear), 5),
                     "probe_tflops": probe,
                     "frac_of_probe_f16": round(gemm_tflops / probe["f16"], 4) if probe else None,
                     "timing": ("value: one CUDA-graph replay per step (selection, pack, quantizer, GEMM), "
                                "no event nodes inside; kernel classes: the step's GEMM (quantizer, "
                                "selection + pack) launches alone, graph-replayed once per timed step "
                                "between two events")
                               if graphs else "eager launches"},
        "weights_select_pack_ms_per_step": round(weights_ms / K_, 4),
        "act_quant": {"achieved_gbs": round(quant_gbs, 1), "peak_gbs": pk["hbm_gbs"],
                      "frac": round(quant_gbs / pk["hbm_gbs"], 4), "ms_per_step": round(quant_ms / K_, 4),
                      "bytes": "2 B read + 2 B fp16 operand write per element"},
        "variants": variants,
        "calibration": route_vs_argmin(cl, lut, cal_sse),
        "gpu_launches": launches * K_,
        "clocks": clocks,
    }
    if not args.no_e2e:
        del X
        result["e2e"] = e2e_leg(args, torch, cl, host, layers, nb, lut, qp, device, stream, world, flops_step)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def e2e_leg(args, torch, cl, host, layers, nb, lut, qp, device, stream, world, flops_step):
    """Same step through the public calls with HOST buffers: the weights and every activation are
    copied host->device from pinned memory and every output device->host inside the timed
    region."""
    import torch.distributed as dist
    Wn, bn, Xn = host
    Wh = [torch.from_numpy(w).pin_memory() for w in Wn]
    bh = [torch.from_numpy(b).pin_memory() for b in bn]
    Xh = [[torch.from_numpy(x).pin_memory() for x in xs] for xs in Xn]
    Yh = [torch.empty((M, N), dtype=torch.float32).pin_memory() for (_, M, K, N) in layers]
    Wd = [w.to(device) for w in Wh]
    bd = [b.to(device) for b in bh]
    Xd = [torch.empty_like(Xh[li][0], device=device) for li in range(len(layers))]
    Yd = [torch.empty((M, N), dtype=torch.float32, device=device) for (_, M, K, N) in layers]
    st = torch.zeros(1, dtype=torch.int32, device=device)
    ws = [torch.empty(max(cl.linear_workspace_size(M, cl.pack_plan(N, K, np.zeros(N, np.uint8)), f)
                          for f in range(6)), dtype=torch.uint8, device=device) for (_, M, K, N) in layers]
    fmt_off = np.cumsum([0] + [N for (_, M, K, N) in layers])
    fmt_all = torch.empty(int(fmt_off[-1]), dtype=torch.uint8, device=device)
    descs = [cl.pack_plan_palette(N, K, cl.PALETTE_W8) for (_, M, K, N) in layers]
    blobs = [torch.empty(d.bytes, dtype=torch.uint8, device=device) for d in descs]
    h2d = sum(w.numel() * 2 + b.numel() * 4 for w, b in zip(Wh, bh)) + sum(x.numel() * 2 for xs in Xh for x in xs)
    d2h = nb * sum(M * N * 4 for (_, M, K, N) in layers)

    # streams for host->device copies, the library calls and (two) device->host copies; per-layer events
    # keep each layer's input and output buffers from being overwritten while still in use, so
    # one layer's upload and download overlap the other layers' compute
    s_h2d = torch.cuda.Stream(device)
    s_d2h_all = [torch.cuda.Stream(device) for _ in range(2)]  # 1 to 6 download streams measured the same
    ev = lambda: [torch.cuda.Event() for _ in layers]
    x_ready, x_free, y_ready, y_free = ev(), ev(), ev(), ev()
    w_ready = torch.cuda.Event()

    def step():
        with torch.cuda.stream(s_h2d):
            for li in range(len(layers)):
                Wd[li].copy_(Wh[li], non_blocking=True)
                bd[li].copy_(bh[li], non_blocking=True)
            w_ready.record(s_h2d)
        stream.wait_event(w_ready)
        for li in range(len(layers)):
            f = fmt_all[fmt_off[li]:fmt_off[li + 1]]
            cl.select_pack_palette(Wd[li], cl.PALETTE_W8, descs[li], fmt_out=f, blob=blobs[li], dev_status=st,
                                   stream=stream)
        for bk in range(nb):
            for li in range(len(layers)):
                with torch.cuda.stream(s_h2d):
                    s_h2d.wait_event(x_free[li])
                    Xd[li].copy_(Xh[li][bk], non_blocking=True)
                    x_ready[li].record(s_h2d)
                stream.wait_event(x_ready[li])
                stream.wait_event(y_free[li])
                cl.linear_static(Xd[li], descs[li], blobs[li], int(lut[li, bk]), qp[li][bk], bias=bd[li], Y=Yd[li],
                                 ws=ws[li], dev_status=st, stream=stream)
                x_free[li].record(stream)
                y_ready[li].record(stream)
                s_d2h = s_d2h_all[li % len(s_d2h_all)]
                with torch.cuda.stream(s_d2h):
                    s_d2h.wait_event(y_ready[li])
                    Yh[li].copy_(Yd[li], non_blocking=True)
                    y_free[li].record(s_d2h)
        for li in range(len(layers)):      # the step ends when its last download has landed
            stream.wait_event(y_free[li])
        # the next step's weight upload must not overwrite weights still read by this step
        s_h2d.wait_stream(stream)

    for e in x_free + y_free:             # a fresh event: waiting on it is a no-op
        e.record(stream)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step()
    t1.record(stream)
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    if world > 1:
        ms = max_over_ranks(ms, device)
    assert int(st.item()) == 0
    return {"value": round(job_tflops(flops_step, args.steps, world, ms), 3), "unit": "TFLOP/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": round(ms / args.steps, 3)}


# ------------------------------------------------------------------ the oracle as CPU baseline
def oracle_sample(layers_idx=(4,), buckets=(0, 5, 9)):
    """The oracle on a bounded sample of the workload: for each (layer, bucket) of the sample,
    per-channel selection over the W8 palette, the pack (codes and scales of the selected formats,
    decoded to their exact values), the activation quantizer in the format the route picks with the
    static scale of the tensor's range (Alg. 1 -> Alg. 2), and the fp64 GEMM over all rows, each
    stage timed.  Returns (flops, seconds, description, seconds per stage)."""
    from oracle import formats as F
    from oracle import gemm as G
    from oracle import schedule as S
    from oracle import select as SEL
    from paper_2609_33496_gb300 import workloads as WL
    snr = S.snr(S.betas_scaled_linear())
    flops, stages = 0.0, {"select": 0.0, "pack": 0.0, "act_quant": 0.0, "gemm": 0.0}
    for li in layers_idx:
        name, M, K, N = WL.SDXL_PROJ_LAYERS[li]
        W, bias = WL.sdxl_layer_weights(li)
        for bk in buckets:
            X = WL.sdxl_layer_activation(li, bk)
            # calibration (the LUT entry and the stored range) is not part of the timed path
            f = S.route(S.kurtosis(X), snr[int(S.bucket_midpoint(bk))])
            x = X.astype(np.float32)
            lo, hi = float(x.min()), float(x.max())
            t0 = time.perf_counter()
            fmt, _, _ = SEL.select_formats(W, 0x007)
            t1 = time.perf_counter()
            a = F.act_dequant(F.act_quant(X, f, lo, hi))
            t2 = time.perf_counter()
            w = SEL.dequant_selected(W, fmt)      # the pack's codes and scales, decoded exactly
            t3 = time.perf_counter()
            G.linear_output(a, w, bias)
            t4 = time.perf_counter()
            stages["select"] += t1 - t0
            stages["act_quant"] += t2 - t1
            stages["pack"] += t3 - t2
            stages["gemm"] += t4 - t3
            flops += layer_flops(M, K, N)
    desc = "oracle select(W8)+pack+static act-quant+fp64 GEMM of layer(s) %s at buckets %s, one BLAS thread" % (
        [WL.SDXL_PROJ_LAYERS[i][0] for i in layers_idx], list(buckets))
    return flops, sum(stages.values()), desc, stages


def variant_matrix(torch, cl, W, bias, X, layers, lut, qp, st, pk, probe, reps=20):
    """Every activation-format x weight-palette variant of the GEMM (plus W4A16) on the largest
    layer of the step, and the quantizer per activation format, the selection and the pack per
    palette on the same tensors.  Each figure is `reps` launches captured in one CUDA graph and
    timed between two events after a warm replay (kernel timed alone: burst peaks apply)."""
    li = max(range(len(layers)), key=lambda i: layer_flops(*layers[i][1:]))
    name, M, K, N = layers[li]
    x = X[li][-1]
    dev = x.device
    Y = torch.empty((M, N), dtype=torch.float32, device=dev)
    hbm = pk["hbm_gbs"] * 1e9
    p16 = (probe or {}).get("f16", pk.get("bf16_tflops", 1900.0)) * 1e12
    p8 = (probe or {}).get("f8f6f4", 2 * p16 / 1e12) * 1e12

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
        return e0.elapsed_time(e1) / reps  # ms per launch

    out = {"layer": name, "M": M, "K": K, "N": N, "reps": reps, "gemm": [], "quant": [], "weights": [],
           "peaks": {"f16_tflops": round(p16 / 1e12, 1), "f8_tflops": round(p8 / 1e12, 1),
                     "hbm_gbs": pk["hbm_gbs"], "source": "tensor-core probe of this run; measured HBM copy"}}
    flops = layer_flops(M, K, N)
    for pal_name, mask, bits in (("W8", cl.PALETTE_W8, 8), ("W4", cl.PALETTE_W4, 4)):
        fmt = torch.empty(N, dtype=torch.uint8, device=dev)
        t_sel = timed(lambda: cl.select_weight_formats(W[li], mask, fmt_out=fmt))
        desc = cl.pack_plan(N, K, fmt.cpu().numpy())
        blob, _ = cl.pack_weights(W[li], fmt, desc, dev_status=st)
        t_pack = timed(lambda: cl.pack_weights(W[li], fmt, desc, dev_status=st, blob=blob))
        pack_bytes = 2 * N * K + N * K * bits / 8 + 10 * N
        t_fused = None
        if mask == cl.PALETTE_W8:   # one MMA class: the fused select + pack of the step
            d_pal = cl.pack_plan_palette(N, K, mask)
            blob_pal = torch.empty(d_pal.bytes, dtype=torch.uint8, device=dev)
            t_fused = timed(lambda: cl.select_pack_palette(W[li], mask, d_pal, fmt_out=fmt, blob=blob_pal,
                                                           dev_status=st))
        out["weights"].append({"palette": pal_name, "select_us": round(t_sel * 1e3, 2),
                               "select_pack_fused_us": None if t_fused is None else round(t_fused * 1e3, 2),
                               "pack_us": round(t_pack * 1e3, 2),
                               "pack_gbs": round(pack_bytes / (t_pack * 1e-3) / 1e9, 1),
                               "pack_frac_hbm": round(pack_bytes / (t_pack * 1e-3) / hbm, 4),
                               "formats": {int(f): int(c) for f, c in zip(*np.unique(fmt.cpu().numpy(),
                                                                                       return_counts=True))}})
        ws = torch.empty(max(cl.linear_workspace_size(M, desc, f) for f in range(6)), dtype=torch.uint8, device=dev)
        for af in ([0, 1, 2, 3, 4] + ([5] if bits == 4 else [])):
            if af != 5:
                cl.linear_prepare(x, desc, af, ws, st)
            t = timed(lambda: cl.linear_gemm(x, desc, blob, af, bias[li], Y, ws, st))
            a_bytes = M * K * (2 if af == 5 else 1) + (M * K / 32 if af in (3, 4) else 0)
            byts = a_bytes + N * K * bits / 8 + 9 * N + 4 * M * N
            t_s = t * 1e-3
            row = {"act_fmt": af, "weights": pal_name, "tflops": round(flops / t_s / 1e12, 1),
                   "us": round(t * 1e3, 2),
                   "frac_f16_roofline": round(max(flops / p16, byts / hbm) / t_s, 4)}
            if af != 5:
                row["frac_fp8_roofline"] = round(max(flops / p8, byts / hbm) / t_s, 4)
            out["gemm"].append(row)
            if bits == 8 and af != 5:
                tq = timed(lambda: cl.linear_prepare(x, desc, af, ws, st))
                xf = x.float()
                p_af = cl.scale_zp(af, float(xf.min()), float(xf.max())) if af <= 2 else None
                tqs = timed(lambda: cl.linear_prepare_static(x, desc, af, p_af, ws, st))
                qb = 4 * M * K
                out["quant"].append({"act_fmt": af, "us": round(tq * 1e3, 2), "static_us": round(tqs * 1e3, 2),
                                     "gbs": round(qb / (tq * 1e-3) / 1e9, 1),
                                     "static_gbs": round(qb / (tqs * 1e-3) / 1e9, 1),
                                     "frac_hbm": round(qb / (tq * 1e-3) / hbm, 4),
                                     "bytes": "2 B read + 2 B fp16 operand write per element"})
    # output type and scale granularity of the epilogue on the largest layer and on the first
    # layer with a large fp32 output (8192 x 640 x 640): f32 / f16 / bf16 Y, one tensor scale or
    # two per-sample scales (the DiT path's), E4M3 activations, W8 weights
    out["epilogue"] = []
    tdt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}
    hbm_layer = next((j for j, l in enumerate(layers) if l[1] >= 8192), None)
    for lj in sorted({li} | ({hbm_layer} if hbm_layer is not None else set())):
        lname, Ml, Kl, Nl = layers[lj]
        desc_l = cl.pack_plan_palette(Nl, Kl, cl.PALETTE_W8)
        fmt_l = torch.empty(Nl, dtype=torch.uint8, device=dev)
        cl.select_weight_formats(W[lj], cl.PALETTE_W8, fmt_out=fmt_l)
        blob_l = torch.empty(desc_l.bytes, dtype=torch.uint8, device=dev)
        cl.pack_weights(W[lj], fmt_l, desc_l, dev_status=st, blob=blob_l)
        ws_l = torch.zeros(cl.linear_workspace_size(Ml, desc_l, 1), dtype=torch.uint8, device=dev)
        fl = layer_flops(Ml, Kl, Nl)
        for groups in (1, 2):
            cl.linear_prepare_groups(X[lj][-1], desc_l, 1, groups, ws_l, st)
            for yn in ("f32", "f16", "bf16"):
                Y_l = torch.empty((Ml, Nl), dtype=tdt[yn], device=dev)
                t = timed(lambda: cl.linear_gemm_ex(X[lj][-1], desc_l, blob_l, 1, groups, bias[lj], Y_l, ws_l,
                                                    st)) * 1e-3
                byts = Ml * Kl + Nl * Kl + 9 * Nl + Y_l.element_size() * Ml * Nl
                out["epilogue"].append({"layer": lname, "y": yn, "groups": groups, "us": round(t * 1e6, 2),
                                        "tflops": round(fl / t / 1e12, 1),
                                        "frac_f16_roofline": round(max(fl / p16, byts / hbm) / t, 4)})
            del Y_l
    # every layer of the step: its GEMM alone in the LUT format of bucket 9, f16 roofline
    # (max(flops / f16 peak, bytes / HBM)) and whether it is tensor- or HBM-bound
    out["layers"] = []
    for lj, (lname, Ml, Kl, Nl) in enumerate(layers):
        af = int(lut[lj, -1])
        desc_l = cl.pack_plan_palette(Nl, Kl, cl.PALETTE_W8)
        fmt_l = torch.empty(Nl, dtype=torch.uint8, device=dev)
        cl.select_weight_formats(W[lj], cl.PALETTE_W8, fmt_out=fmt_l)
        blob_l = torch.empty(desc_l.bytes, dtype=torch.uint8, device=dev)
        cl.pack_weights(W[lj], fmt_l, desc_l, dev_status=st, blob=blob_l)
        ws_l = torch.zeros(cl.linear_workspace_size(Ml, desc_l, af), dtype=torch.uint8, device=dev)
        Y_l = torch.empty((Ml, Nl), dtype=torch.float32, device=dev)
        cl.linear_prepare_static(X[lj][-1], desc_l, af, qp[lj][-1], ws_l, st)
        t = timed(lambda: cl.linear_gemm(X[lj][-1], desc_l, blob_l, af, bias[lj], Y_l, ws_l, st)) * 1e-3
        fl = layer_flops(Ml, Kl, Nl)
        byts = Ml * Kl + Nl * Kl + 9 * Nl + 4 * Ml * Nl
        t_f, t_b = fl / p16, byts / hbm
        out["layers"].append({"layer": lname, "M": Ml, "K": Kl, "N": Nl, "act_fmt": af, "us": round(t * 1e6, 2),
                              "tflops": round(fl / t / 1e12, 1), "bound": "tensor" if t_f >= t_b else "hbm",
                              "frac_f16_roofline": round(max(t_f, t_b) / t, 4)})
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "device status %d" % int(st.item())
    return out


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


def dit_sampler(torch, cl, st, steps=20):
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
    M = 128, N = 192, on seeded finite operands.  Returns TFLOP/s per kind."""
    import ctypes
    from paper_2609_33496_gb300 import build as B
    L = ctypes.CDLL(B.PROBE_LIB)
    L.chameleon_probe_mma.argtypes = [ctypes.c_int] * 4 + [ctypes.c_void_p] * 3
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    cyc = torch.zeros(1, dtype=torch.int64, device=device)
    st = torch.zeros(1, dtype=torch.int32, device=device)
    s = torch.cuda.current_stream()
    out = {}
    for kind, name, K in ((0, "f16", 16), (2, "f8f6f4", 32)):
        iters, best = 4000, 0.0
        for _ in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            rc = L.chameleon_probe_mma(kind, 192, sms, iters, ctypes.c_void_p(cyc.data_ptr()),
                                       ctypes.c_void_p(st.data_ptr()), ctypes.c_void_p(s.cuda_stream))
            e1.record(s)
            torch.cuda.synchronize()
            if rc != 0 or int(st.item()) != 0:
                return None
            best = max(best, sms * iters * 4 * 2.0 * 128 * 192 * K / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        out[name] = round(best, 1)
    return out


def cpu_baseline():
    # one core: the BLAS and OpenMP pools of this process are limited to one thread at start-up
    # about ten seconds of one Grace core: two layers (q and FF-out) at five buckets
    flops, t, desc, stages = oracle_sample(layers_idx=(4, 9), buckets=(0, 3, 5, 7, 9))
    return {"value": round(flops / t / 1e12, 6), "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
            "sample": desc, "seconds": round(t, 2), "stage_seconds": {k: round(v, 3) for k, v in stages.items()},
            "host_cores": os.cpu_count()}


def reference_arm(args, world):
    for _ in range(args.warmup):
        oracle_sample(buckets=(9,))
    flops, t = 0.0, 0.0
    desc = ""
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


if __name__ == "__main__":
    sys.exit(main())

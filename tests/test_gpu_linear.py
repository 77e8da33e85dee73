"""GPU quantized linear (a7, a8) against the fp64 oracle on the same dequantized operands:
|Y - Y_ref| <= 2^-10 * sum_k |a_k w_k| per element."""
import numpy as np
import pytest

from oracle import formats as F
from oracle import gemm as G
from oracle import select as SEL
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host, assert_within_bound

pytestmark = pytest.mark.gpu
ACT = [F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2, F.A_MXFP8, F.A_MXINT8]


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def gpu_linear(cl, X, W, fmt, act_fmt, bias, f16_only=0, layout=0, fold=0):
    import torch
    d = cl.pack_plan(W.shape[0], W.shape[1], fmt, layout, fold)
    d.f16_only = f16_only
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    Y, st2 = cl.linear(cuda(X), d, blob, act_fmt, bias=None if bias is None else cuda(bias))
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st2.item()) == 0
    return host(Y)


def check(cl, X, W, fmt, act_fmt, bias, what, f16_only=0):
    Y = gpu_linear(cl, X, W, fmt, act_fmt, bias, f16_only)
    Y_ref, bound, _, _ = G.linear_reference(X, act_fmt, W, fmt, bias)
    assert_within_bound(Y, Y_ref, bound, what)


@pytest.mark.parametrize("f16_only", [0, 1])
@pytest.mark.parametrize("act_fmt", ACT)
@pytest.mark.parametrize("mask", [0x007, 0x1F8])
def test_single_layer_w8a8_w4a8(cl, act_fmt, mask, f16_only):
    """Config 1; with f16_only = 0 the 4-bit class-0 tiles run on FP8 MMAs for E4M3 / E5M2 / MXFP8
    activations, with 1 every tile runs on fp16 MMAs."""
    X, W, bias = WL.single_layer()
    fmt, _, _ = SEL.select_formats(W, mask)
    check(cl, X, W, fmt, act_fmt, bias, "act %d mask %#x f16_only %d" % (act_fmt, mask, f16_only), f16_only)


def test_weight_only_fp16_activations(cl):
    X, W, bias = WL.single_layer()
    fmt, _, _ = SEL.select_formats(W, 0x1F8)
    check(cl, X, W, fmt, F.A_FP16, bias, "W4A16")


@pytest.mark.parametrize("M,K,N", [(1, 32, 1), (2, 96, 130), (17, 160, 129), (200, 64, 300),
                                   (300, 320, 257), (130, 352, 64)])
@pytest.mark.parametrize("bits,f16_only", [(8, 0), (4, 0), (4, 1)])
def test_ragged_shapes_every_format(cl, M, K, N, bits, f16_only):
    g = np.random.default_rng(M * 1000 + K + N)
    X = WL.to_fp16(g.standard_t(4, (M, K)))
    W = WL.weight_mix(g, N, K)
    pal = F.W8_PALETTE if bits == 8 else F.W4_PALETTE
    fmt = np.asarray(pal, np.uint8)[g.integers(0, len(pal), N)]
    bias = g.normal(0, 0.02, N).astype(np.float32)
    for act_fmt in ACT + [F.A_FP16]:
        check(cl, X, W, fmt, act_fmt, bias if act_fmt % 2 else None,
              "M%d K%d N%d bits %d act %d f16_only %d" % (M, K, N, bits, act_fmt, f16_only), f16_only)


@pytest.mark.parametrize("fold", [0, 48])
@pytest.mark.parametrize("M,K,N", [(17, 160, 300), (300, 352, 500)])
def test_format_group_layout_every_activation(cl, M, K, N, fold):
    """The format-group layout (one format per tile, small formats folded into a class tail) gives
    the same bound on every activation format, on the FP8 and the fp16 paths."""
    g = np.random.default_rng(M + K + N + fold)
    X = WL.to_fp16(g.standard_t(4, (M, K)))
    W = WL.weight_mix(g, N, K)
    fmt = np.asarray(F.W4_PALETTE, np.uint8)[g.choice(len(F.W4_PALETTE), N, p=[0.1, 0.3, 0.2, 0.05, 0.05, 0.3])]
    bias = g.normal(0, 0.02, N).astype(np.float32)
    for act_fmt in ACT + [F.A_FP16]:
        Y = gpu_linear(cl, X, W, fmt, act_fmt, bias, layout=1, fold=fold)
        Y_ref, bound, _, _ = G.linear_reference(X, act_fmt, W, fmt, bias)
        assert_within_bound(Y, Y_ref, bound, "layout 1 fold %d act %d" % (fold, act_fmt))


@pytest.mark.parametrize("M", [1, 2, 8, 16])
@pytest.mark.parametrize("K,N", [(320, 1280), (1280, 1280), (2048, 640)])
def test_small_m_weight_streaming(cl, M, K, N):
    """Up to 16 tokens the weight-streaming kernel runs (one cluster of K ranges per 64 channels):
    the few-step fork's weight-only rows (SDXL-Turbo shapes at batch 1 to 16) with the mixed 4-bit
    formats, the 8-bit palette with INT8-asym and MXFP8 activations, every element within the bound."""
    g = np.random.default_rng(M * 7 + K + N)
    X = WL.to_fp16(g.standard_t(4, (M, K)) * np.exp(0.1 * g.standard_normal(K))[None, :])
    W = WL.weight_mix(g, N, K)
    bias = g.normal(0, 0.02, N).astype(np.float32)
    for pal, acts in ((F.W4_PALETTE, [F.A_FP16, F.A_E4M3]), (F.W8_PALETTE, [F.A_INT8_ASYM, F.A_MXFP8])):
        fmt = np.asarray(pal, np.uint8)[g.integers(0, len(pal), N)]
        for act_fmt in acts:
            check(cl, X, W, fmt, act_fmt, bias, "small M%d K%d N%d act %d" % (M, K, N, act_fmt))


def test_small_m_output_types_groups_and_group_wise_weights(cl):
    """The weight-streaming kernel's epilogue: fp16 / bf16 outputs (the fp32 value rounded once),
    two per-sample scales, and a group-wise blob (fp16 group scales in the decode)."""
    import torch
    g = np.random.default_rng(41)
    M, K, N = 16, 640, 384
    X = WL.to_fp16(g.standard_t(5, (M, K)))
    W = WL.weight_mix(g, N, K)
    fmt = np.asarray(F.W4_PALETTE, np.uint8)[g.integers(0, 6, N)]
    d = cl.pack_plan(N, K, fmt)
    blob, _ = cl.pack_weights(cuda(W), cuda(fmt), d)
    for y_dtype in (torch.float32, torch.float16, torch.bfloat16):
        Y, st = cl.linear_ex(cuda(X), d, blob, F.A_E5M2, n_groups=2, y_dtype=y_dtype)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        qs = F.act_quant_per_sample(X, F.A_E5M2, 2)
        a = F.act_dequant_per_sample(qs)
        y_ref, bound = G.linear_rows_reference(a, SEL.dequant_selected(W, fmt), np.arange(M))
        y = host(Y.float())
        half = 0 if y_dtype == torch.float32 else np.abs(y_ref) * (2.0 ** -11 if y_dtype == torch.float16 else 2.0 ** -8)
        assert_within_bound(y, y_ref, bound + half, "small M per-sample %s" % y_dtype)
    dg = cl.pack_plan_grouped(N, K, F.W_INT4_ASYM, 64)
    bg, _ = cl.pack_weights(cuda(W), cuda(np.full(N, F.W_INT4_ASYM, np.uint8)), dg)
    Y, st = cl.linear(cuda(X), dg, bg, F.A_FP16)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    wq = SEL.grouped_dequant(W, 64, F.W_INT4_ASYM)
    y_ref, bound = G.linear_rows_reference(X.astype(np.float64), wq, np.arange(M))
    assert_within_bound(host(Y), y_ref, bound, "small M group-wise")


CLASS0 = [F.W_INT4_SYM, F.W_INT4_ASYM, F.W_E2M1, F.W_MXINT4, F.W_MXFP4]


@pytest.mark.parametrize("wfmt", CLASS0)
@pytest.mark.parametrize("act_fmt", [F.A_E4M3, F.A_E5M2, F.A_MXFP8])
@pytest.mark.parametrize("M,K,N", [(300, 352, 300), (161, 4608, 129)])
def test_fp8_path_every_activation_weight_pair(cl, act_fmt, wfmt, M, K, N):
    """Each FP8 activation format x each class-0 weight format on the 8-bit tensor cores
    (kind::mxf8f6f4): several channel and token tiles, a ragged last K-chunk (352 = 2 x 128 + 3
    blocks of 32, the last 64-element blob chunk alone) and a long K; every channel in one format,
    MX weights with block exponents that vary along K (outlier channels, mixed distributions)."""
    g = np.random.default_rng(7 * M + K + N + 13 * wfmt + act_fmt)
    X = WL.to_fp16(g.standard_t(5, (M, K)) * np.exp(0.1 * g.standard_normal(K))[None, :])
    W = WL.weight_mix(g, N, K)
    fmt = np.full(N, wfmt, np.uint8)
    bias = g.normal(0, 0.02, N).astype(np.float32)
    check(cl, X, W, fmt, act_fmt, bias, "act %d w %d M%d K%d N%d" % (act_fmt, wfmt, M, K, N))


def test_exact_special_operands(cl):
    """W = I in MXINT8 (DQ exactly I): Y equals DQ(A) exactly; zero rows give exactly the bias."""
    K = 128
    X = WL.to_fp16(np.random.default_rng(2).standard_t(3, (64, K)))
    X[5] = 0
    W = np.eye(K, dtype=np.float16)
    fmt = np.full(K, F.W_MXINT8, np.uint8)
    bias = np.random.default_rng(3).normal(0, 1, K).astype(np.float32)
    for act_fmt in ACT:
        Y = gpu_linear(cl, X, W, fmt, act_fmt, bias)
        a = F.act_dequant(F.act_quant(X, act_fmt))
        np.testing.assert_array_equal(Y, (a + bias[None, :]).astype(np.float32))


def test_deterministic(cl):
    X, W, bias = WL.single_layer()
    fmt, _, _ = SEL.select_formats(W, 0x1F8)
    Y1 = gpu_linear(cl, X, W, fmt, F.A_E4M3, bias)
    Y2 = gpu_linear(cl, X, W, fmt, F.A_E4M3, bias)
    assert Y1.tobytes() == Y2.tobytes()


@pytest.mark.parametrize("layer", range(len(WL.SDXL_PROJ_LAYERS)))
def test_full_size_sdxl_projection_sampled_rows(cl, layer):
    """Full-size W8A8 SDXL projections in the launch configuration the benchmark uses; the fp64
    reference is computed on 96 seeded rows."""
    import torch
    name, M, K, N = WL.SDXL_PROJ_LAYERS[layer]
    W, bias = WL.sdxl_layer_weights(layer)
    fmt_dev, _ = cl.select_weight_formats(cuda(W), 0x007)
    fmt = host(fmt_dev)
    for bucket, act_fmt in [(9, F.A_E5M2), (3, F.A_E4M3), (0, F.A_INT8_ASYM)]:
        X = WL.sdxl_layer_activation(layer, bucket)
        Y = gpu_linear(cl, X, W, fmt, act_fmt, bias)
        rows = np.sort(np.random.default_rng(layer).choice(M, 96, replace=False))
        a = F.act_dequant(F.act_quant(X, act_fmt))
        w = SEL.dequant_selected(W, fmt)
        y_ref, bound = G.linear_rows_reference(a, w, rows, bias)
        assert_within_bound(Y[rows], y_ref, bound, "%s bucket %d" % (name, bucket))


W4_TURBO = (1 << F.W_INT4_ASYM) | (1 << F.W_NF4) | (1 << F.W_E2M1) | (1 << F.W_MXINT4) | (1 << F.W_MXFP4)
WIDE_CASES = ([(3, i, shp, [F.A_E4M3, F.A_E5M2]) for i, shp in enumerate(WL.UNET_W4A8_SHAPES)]
              + [(4, i, shp, [F.A_E4M3, F.A_MXFP8]) for i, shp in enumerate(WL.PIXART_W4A8_SHAPES)]
              + [(5, i, shp, [F.A_FP16]) for i, shp in enumerate(WL.TURBO_W4A16_SHAPES)])


@pytest.mark.parametrize("config,index,shape,act_fmts", WIDE_CASES)
def test_wider_workload_shapes_sampled_rows(cl, config, index, shape, act_fmts):
    """SDXL-UNet and PixArt-alpha W4A8 layers and SDXL-Turbo W4A16 layers (M from 1 to 32768)
    with the 4-bit palette of those workloads selected on the GPU; the fp64 reference is computed
    on up to 64 seeded rows."""
    M, K, N = shape
    X, W, bias = WL.config_layer(config, index, M, K, N)
    fmt_dev, _ = cl.select_weight_formats(cuda(W), W4_TURBO)
    fmt = host(fmt_dev)
    w = SEL.dequant_selected(W, fmt)
    rows = np.arange(M) if M <= 64 else np.sort(np.random.default_rng(index).choice(M, 64, replace=False))
    for act_fmt in act_fmts:
        Y = gpu_linear(cl, X, W, fmt, act_fmt, bias)
        a = X.astype(np.float64) if act_fmt == F.A_FP16 else F.act_dequant(F.act_quant(X, act_fmt))
        y_ref, bound = G.linear_rows_reference(a, w, rows, bias)
        assert_within_bound(Y[rows], y_ref, bound, "config %d %s act %d" % (config, shape, act_fmt))

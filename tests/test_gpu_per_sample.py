"""GPU per-sample activation scales (Alg. 3 with the range of each sample: rows in equal groups)
and fp16 / bf16 outputs of the linear, against the oracle's act_quant_per_sample."""
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


def torch_dtype(name):
    import torch
    return {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[name]


def to_host(Y):
    import torch
    return Y.float().cpu().numpy() if Y.dtype == torch.bfloat16 else host(Y)


def samples(M, K, n_groups, seed):
    """Samples of very different magnitude, so that per-sample and per-tensor scales differ."""
    g = np.random.default_rng(seed)
    R = M // n_groups
    mag = 2.0 ** g.integers(-4, 5, n_groups)
    return WL.to_fp16(np.vstack([g.standard_t(4, (R, K)) * mag[i] for i in range(n_groups)]))


@pytest.mark.parametrize("act_fmt", ACT)
@pytest.mark.parametrize("M,n_groups", [(64, 1), (64, 4), (60, 4), (300, 3), (256, 64)])
def test_identity_weights_give_the_per_sample_dequantized_operand_exactly(cl, act_fmt, M, n_groups):
    """W = I in MXINT8 (DQ exactly I): each output row equals that row's per-sample dequantized
    activation plus the bias, rounded once to fp32 -- checks every group's scale and zero point
    bit for bit, including groups that end inside a 16-token slice (15 rows) or a tile."""
    import torch
    K = 128
    X = samples(M, K, n_groups, M + n_groups)
    W = np.eye(K, dtype=np.float16)
    fmt = np.full(K, F.W_MXINT8, np.uint8)
    bias = np.random.default_rng(3).normal(0, 1, K).astype(np.float32)
    d = cl.pack_plan(K, K, fmt)
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    Y, st2 = cl.linear_ex(cuda(X), d, blob, act_fmt, n_groups, bias=cuda(bias))
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st2.item()) == 0
    a = F.act_dequant_per_sample(F.act_quant_per_sample(X, act_fmt, n_groups))
    np.testing.assert_array_equal(host(Y), (a + bias[None, :]).astype(np.float32))


@pytest.mark.parametrize("y", ["f16", "bf16"])
def test_identity_weights_half_outputs_round_the_fp32_value(cl, y):
    """fp16 / bf16 outputs are the fp32 value rounded to nearest even (values beyond fp16's range
    become +-Inf)."""
    import torch
    K = 64
    X = samples(32, K, 2, 5)
    X[3, 7] = np.float16(60000.0)
    W = np.eye(K, dtype=np.float16)
    fmt = np.full(K, F.W_MXINT8, np.uint8)
    bias = np.zeros(K, np.float32)
    bias[7] = 30000.0
    d = cl.pack_plan(K, K, fmt)
    blob, _ = cl.pack_weights(cuda(W), cuda(fmt), d)
    Y, st = cl.linear_ex(cuda(X), d, blob, F.A_E5M2, 2, y_dtype=torch_dtype(y), bias=cuda(bias))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    y32 = (F.act_dequant_per_sample(F.act_quant_per_sample(X, F.A_E5M2, 2)) + bias[None, :]).astype(np.float32)
    if y == "f16":
        ref = y32.astype(np.float16)
        assert np.isinf(ref[3, 7])
        np.testing.assert_array_equal(host(Y), ref)
    else:
        ref = torch.from_numpy(y32).to(torch.bfloat16).float().numpy()
        np.testing.assert_array_equal(to_host(Y), ref)


def check_rows(Y, y_ref, bound, y, what):
    """fp32: within the accumulation bound; fp16 / bf16: plus half a unit in the last place of the
    output type at the fp32 value (and the smallest subnormal spacing for fp16)."""
    if y == "f32":
        assert_within_bound(Y, y_ref, bound, what)
        return
    u = 2.0 ** -11 if y == "f16" else 2.0 ** -8
    tiny = 2.0 ** -25 if y == "f16" else 0.0
    tol = bound + u * (np.abs(y_ref) + bound) + tiny
    err = np.abs(Y.astype(np.float64) - y_ref)
    bad = err > tol
    assert not bad.any(), "%s: %d outputs outside the bound, worst %g" % (what, int(bad.sum()), float((err - tol).max()))


@pytest.mark.parametrize("act_fmt", [F.A_INT8_ASYM, F.A_E4M3, F.A_MXFP8])
@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("y", ["f32", "f16", "bf16"])
def test_per_sample_linear_matches_oracle(cl, act_fmt, bits, y):
    import torch
    g = np.random.default_rng(60 + act_fmt * 7 + bits)
    M, K, N, n_groups = 300, 320, 257, 5
    X = samples(M, K, n_groups, 61 + bits)
    W = WL.weight_mix(g, N, K)
    pal = F.W8_PALETTE if bits == 8 else F.W4_PALETTE
    fmt = np.asarray(pal, np.uint8)[g.integers(0, len(pal), N)]
    bias = g.normal(0, 0.02, N).astype(np.float32)
    d = cl.pack_plan(N, K, fmt)
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    Y, st2 = cl.linear_ex(cuda(X), d, blob, act_fmt, n_groups, y_dtype=torch_dtype(y), bias=cuda(bias))
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st2.item()) == 0
    a = F.act_dequant_per_sample(F.act_quant_per_sample(X, act_fmt, n_groups))
    y_ref, bound = G.linear_rows_reference(a, SEL.dequant_selected(W, fmt), np.arange(M), bias)
    check_rows(to_host(Y), y_ref, bound, y, "act %d bits %d %s" % (act_fmt, bits, y))


@pytest.mark.parametrize("index", range(len(WL.PIXART_W4A8_SHAPES)))
def test_pixart_shapes_two_samples_sampled_rows(cl, index):
    """PixArt-alpha W4A8 layers with the batch's two samples scaled separately (the DiT path) and
    fp16 outputs; fp64 reference on 64 seeded rows."""
    import torch
    M, K, N = WL.PIXART_W4A8_SHAPES[index]
    n_groups = 2 if M % 2 == 0 else 1
    X, W, bias = WL.config_layer(4, index, M, K, N)
    R = M // n_groups
    X[R:] = (X[R:].astype(np.float32) * 4.0).astype(np.float16)   # the second sample 4x larger
    fmt_dev, _ = cl.select_weight_formats(cuda(W), (1 << F.W_INT4_ASYM) | (1 << F.W_E2M1) | (1 << F.W_MXFP4))
    fmt = host(fmt_dev)
    d = cl.pack_plan(N, K, fmt)
    blob, st = cl.pack_weights(cuda(W), fmt_dev, d)
    w = SEL.dequant_selected(W, fmt)
    rows = np.arange(M) if M <= 64 else np.sort(np.random.default_rng(index).choice(M, 64, replace=False))
    for act_fmt in (F.A_E5M2, F.A_E4M3):
        Y, st2 = cl.linear_ex(cuda(X), d, blob, act_fmt, n_groups, y_dtype=torch.float16, bias=cuda(bias))
        torch.cuda.synchronize()
        assert int(st.item()) == 0 and int(st2.item()) == 0
        qs = F.act_quant_per_sample(X, act_fmt, n_groups)
        a = np.vstack([F.act_dequant(q) for q in qs])
        y_ref, bound = G.linear_rows_reference(a, w, rows, bias)
        check_rows(host(Y)[rows], y_ref, bound, "f16", "%s act %d" % ((M, K, N), act_fmt))


@pytest.mark.parametrize("act_fmt", [F.A_E4M3, F.A_INT8_ASYM, F.A_MXFP8])
def test_chained_linears_read_the_previous_output(cl, act_fmt):
    """One linear's fp16 output fed straight to the next linear on the same stream: the second
    quantizer (launched while the first GEMM may still run) must see the finished output.  The
    output buffer starts filled with 2^14 so that an early read would change the range."""
    import torch
    rng = np.random.default_rng(70 + act_fmt)
    M, K1, K2, N2 = 256, 320, 640, 257
    X = WL.to_fp16(rng.standard_t(4, (M, K1)))
    W1 = WL.weight_mix(rng, K2, K1)
    W2 = WL.weight_mix(rng, N2, K2)
    f1 = np.asarray(F.W8_PALETTE, np.uint8)[rng.integers(0, 3, K2)]
    f2 = np.asarray(F.W8_PALETTE, np.uint8)[rng.integers(0, 3, N2)]
    d1, d2 = cl.pack_plan(K2, K1, f1), cl.pack_plan(N2, K2, f2)
    b1, _ = cl.pack_weights(cuda(W1), cuda(f1), d1)
    b2, _ = cl.pack_weights(cuda(W2), cuda(f2), d2)
    torch.cuda.synchronize()
    Y1 = torch.full((M, K2), 16384.0, dtype=torch.float16, device="cuda")
    for _ in range(3):
        Y1.fill_(16384.0)
        cl.linear_ex(cuda(X), d1, b1, F.A_E4M3, 1, Y=Y1)
        Y2, st = cl.linear_ex(Y1, d2, b2, act_fmt, 2)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        y1 = host(Y1)
        a = F.act_dequant_per_sample(F.act_quant_per_sample(y1, act_fmt, 2))
        y_ref, bound = G.linear_rows_reference(a, SEL.dequant_selected(W2, f2), np.arange(M), None)
        assert_within_bound(host(Y2), y_ref, bound, "chained act %d" % act_fmt)

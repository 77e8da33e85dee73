"""GPU static-scale path (Alg. 2: per-tensor (s, z) fixed beforehand from the calibration range
that Alg. 1 stored for the layer and bucket) against the oracle's act_quant(X, fmt, lo, hi):
codes bit-exact, stored parameters bit-exact, linear outputs within the fp32-accumulation bound."""
import numpy as np
import pytest

from oracle import formats as F
from oracle import gemm as G
from oracle import select as SEL
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host, assert_within_bound

pytestmark = pytest.mark.gpu
TENSOR = [F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2]


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def static_codes(cl, X, fmt, lo, hi):
    import torch
    M, K = X.shape
    p = cl.scale_zp(fmt, lo, hi) if fmt <= F.A_E5M2 else None
    qact, st = cl.act_quant_static(cuda(X), fmt, p)
    torch.cuda.synchronize()
    codes, params, e8 = cl.split_qact(qact, M, K)
    return host(codes), params, host(e8), int(st.item())


def ranges_for(X, g):
    """Calibration ranges around X's own: narrower (clamps), wider, one-sided, degenerate."""
    x = X.astype(np.float32)
    lo, hi = float(x.min()), float(x.max())
    return [(lo, hi), (0.5 * lo, 0.25 * hi), (2.0 * lo, 3.0 * hi), (0.0, hi), (lo, 0.0), (0.0, 0.0),
            (float(np.float32(lo * g.uniform(0.1, 1.5))), float(np.float32(hi * g.uniform(0.1, 1.5))))]


@pytest.mark.parametrize("fmt", TENSOR)
@pytest.mark.parametrize("shape", [(1, 32), (3, 64), (257, 96), (1000, 4096)])
def test_static_codes_match_oracle(cl, fmt, shape):
    g = np.random.default_rng(shape[0] * 7 + shape[1])
    X = WL.to_fp16(g.standard_t(3, shape) * 2.0 ** g.integers(-6, 6))
    for lo, hi in ranges_for(X, g):
        codes, params, _, st = static_codes(cl, X, fmt, lo, hi)
        ref = F.act_quant(X, fmt, lo, hi)
        assert st == 0
        bad = np.argwhere(codes != ref["codes"])
        assert len(bad) == 0, "fmt %d range [%g, %g]: %d codes differ, first at %s" % (fmt, lo, hi, len(bad),
                                                                                     tuple(bad[0]))
        assert np.float32(params["s"]).tobytes() == np.float32(ref["s"]).tobytes()
        assert params["z"] == ref["z"] and params["fmt"] == fmt


@pytest.mark.parametrize("fmt", TENSOR)
def test_static_with_own_range_is_the_dynamic_path(cl, fmt):
    X, _, _ = WL.single_layer()
    x = X.astype(np.float32)
    codes, params, _, _ = static_codes(cl, X, fmt, float(x.min()), float(x.max()))
    qact, _ = cl.act_quant(cuda(X), fmt)
    dyn, dparams, _ = cl.split_qact(qact, *X.shape)
    np.testing.assert_array_equal(codes, host(dyn))
    assert (params["s"], params["z"], params["inv"]) == (dparams["s"], dparams["z"], dparams["inv"])


@pytest.mark.parametrize("fmt", [F.A_MXFP8, F.A_MXINT8])
def test_mx_formats_ignore_static_parameters(cl, fmt):
    X, _, _ = WL.single_layer()
    codes, _, e8, st = static_codes(cl, X, fmt, -1.0, 1.0)
    ref = F.act_quant(X, fmt)
    assert st == 0
    np.testing.assert_array_equal(codes, ref["codes"])
    np.testing.assert_array_equal(e8, ref["e8m0"])


@pytest.mark.parametrize("fmt", TENSOR)
def test_static_nonfinite_input_sets_status(cl, fmt):
    X = WL.to_fp16(np.random.default_rng(1).standard_normal((64, 256)))
    X[17, 100] = np.float16(np.inf) if fmt != F.A_E4M3 else np.float16(np.nan)
    _, _, _, st = static_codes(cl, X, fmt, -4.0, 4.0)
    assert st == cl.ERR_NONFINITE


@pytest.mark.parametrize("act_fmt", TENSOR + [F.A_MXFP8])
@pytest.mark.parametrize("bits", [8, 4])
def test_static_linear_matches_oracle(cl, act_fmt, bits):
    import torch
    g = np.random.default_rng(40 + act_fmt + bits)
    M, K, N = 300, 320, 257
    X = WL.to_fp16(g.standard_t(4, (M, K)))
    W = WL.weight_mix(g, N, K)
    pal = F.W8_PALETTE if bits == 8 else F.W4_PALETTE
    fmt = np.asarray(pal, np.uint8)[g.integers(0, len(pal), N)]
    bias = g.normal(0, 0.02, N).astype(np.float32)
    d = cl.pack_plan(N, K, fmt)
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    x = X.astype(np.float32)
    for lo, hi in [(0.6 * float(x.min()), 0.6 * float(x.max())), (2 * float(x.min()), 1.5 * float(x.max()))]:
        p = cl.scale_zp(act_fmt, lo, hi) if act_fmt <= F.A_E5M2 else None
        Y, st2 = cl.linear_static(cuda(X), d, blob, act_fmt, p, bias=cuda(bias))
        torch.cuda.synchronize()
        assert int(st.item()) == 0 and int(st2.item()) == 0
        a = F.act_dequant(F.act_quant(X, act_fmt, lo, hi))
        w = SEL.dequant_selected(W, fmt)
        y_ref, bound = G.linear_rows_reference(a, w, np.arange(M), bias)
        assert_within_bound(host(Y), y_ref, bound, "act %d bits %d range [%g, %g]" % (act_fmt, bits, lo, hi))


@pytest.mark.parametrize("layer", [0, 3])
def test_full_size_sdxl_static_sampled_rows(cl, layer):
    """Full-size SDXL projections on the static path with scales from a calibration range taken on
    another seeded activation of the same layer and bucket; fp64 reference on 96 seeded rows."""
    import torch
    name, M, K, N = WL.SDXL_PROJ_LAYERS[layer]
    W, bias = WL.sdxl_layer_weights(layer)
    fmt_dev, _ = cl.select_weight_formats(cuda(W), 0x007)
    fmt = host(fmt_dev)
    d = cl.pack_plan(N, K, fmt)
    blob, st = cl.pack_weights(cuda(W), fmt_dev, d)
    w = SEL.dequant_selected(W, fmt)
    for bucket, act_fmt in [(9, F.A_E5M2), (3, F.A_E4M3), (0, F.A_INT8_ASYM)]:
        X = WL.sdxl_layer_activation(layer, bucket)
        xc = WL.sdxl_layer_activation(layer, (bucket + 1) % 10).astype(np.float32)
        lo, hi = float(xc.min()), float(xc.max())
        Y, st2 = cl.linear_static(cuda(X), d, blob, act_fmt, cl.scale_zp(act_fmt, lo, hi), bias=cuda(bias))
        torch.cuda.synchronize()
        assert int(st.item()) == 0 and int(st2.item()) == 0
        rows = np.sort(np.random.default_rng(layer).choice(M, 96, replace=False))
        a = F.act_dequant(F.act_quant(X[rows], act_fmt, lo, hi))
        y_ref, bound = G.linear_rows_reference(a, w, np.arange(len(rows)), bias)
        assert_within_bound(host(Y)[rows], y_ref, bound, "%s bucket %d" % (name, bucket))


def test_check_returns_the_device_status(cl):
    """chameleon_check synchronises and hands back the first device-detected error."""
    import torch
    X = WL.to_fp16(np.random.default_rng(2).standard_normal((64, 256)))
    _, st = cl.act_quant_static(cuda(X), F.A_E4M3, cl.scale_zp(F.A_E4M3, -4.0, 4.0))
    assert cl.device_status(st) == 0
    X[3, 3] = np.float16(np.nan)
    _, st = cl.act_quant_static(cuda(X), F.A_E4M3, cl.scale_zp(F.A_E4M3, -4.0, 4.0))
    assert cl.device_status(st) == cl.ERR_NONFINITE
    assert cl.lib().chameleon_check(None, None) == cl.ERR_INVALID_ARG

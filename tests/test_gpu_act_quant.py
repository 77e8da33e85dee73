"""GPU activation quantizer (steps a2-a4) against the oracle: codes, scales, zero points and E8M0
exponents bit-exact on the same seeded inputs."""
import numpy as np
import pytest

from oracle import formats as F
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host

pytestmark = pytest.mark.gpu
FORMATS = [F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2, F.A_MXFP8, F.A_MXINT8]


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def run(cl, X, fmt):
    import torch
    M, K = X.shape
    qact, st = cl.act_quant(cuda(X), fmt)
    torch.cuda.synchronize()
    codes, params, e8 = cl.split_qact(qact, M, K)
    return host(codes), params, host(e8), int(st.item())


def compare(cl, X, fmt):
    codes, params, e8, st = run(cl, X, fmt)
    ref = F.act_quant(X, fmt)
    assert st == 0
    if not np.array_equal(codes, ref["codes"]):
        bad = np.argwhere(codes != ref["codes"])
        i = tuple(bad[0])
        raise AssertionError("fmt %d: %d codes differ, first at %s: x=%r gpu=%#x ref=%#x"
                             % (fmt, len(bad), i, float(X[i]), codes[i], ref["codes"][i]))
    if fmt <= F.A_E5M2:
        assert np.float32(params["s"]).tobytes() == np.float32(ref["s"]).tobytes()
        assert params["z"] == ref["z"]
        assert params["fmt"] == fmt
    else:
        np.testing.assert_array_equal(e8, ref["e8m0"])


@pytest.mark.parametrize("fmt", FORMATS)
def test_single_layer_workload(cl, fmt):
    X, _, _ = WL.single_layer()
    compare(cl, X, fmt)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("shape", [(1, 32), (3, 64), (257, 96), (1000, 4096)])
def test_ragged_and_multi_cta_shapes(cl, fmt, shape):
    g = np.random.default_rng(hash(shape) % 1000)
    X = WL.to_fp16(g.standard_t(3, shape) * 2.0 ** g.integers(-12, 8))
    compare(cl, X, fmt)


@pytest.mark.parametrize("fmt", FORMATS)
def test_degenerate_inputs(cl, fmt):
    K = 64
    cases = [np.zeros((4, K)), np.full((4, K), -0.0), np.full((4, K), 3.5),
             np.eye(4, K) * -2.0, np.full((2, K), 65504.0), np.full((2, K), 2.0 ** -24)]
    ext = np.zeros((4, K))
    ext[0, :] = 2.0 ** np.arange(-24, -24 + K) % 60000      # wide dynamic range
    ext[1, ::3] = -65504.0
    ext[2, :] = np.linspace(-1e-7, 1e-7, K)
    cases.append(ext)
    for X in cases:
        compare(cl, WL.to_fp16(X), fmt)


@pytest.mark.parametrize("fmt", FORMATS)
def test_rounding_ties_and_saturation(cl, fmt):
    """Values on and near the grid midpoints of every format (the rounding decides)."""
    g = np.random.default_rng(11)
    base = np.concatenate([np.arange(-300, 301) * 0.25, g.standard_t(2, 1399) * 40])
    X = WL.to_fp16(np.resize(base, (16, 128)))
    compare(cl, X, fmt)


def test_nonfinite_sets_status(cl):
    for fmt in FORMATS:
        X = np.ones((8, 64), np.float16)
        X[3, 5] = np.inf if fmt % 2 else np.nan
        _, _, _, st = run(cl, X, fmt)
        assert st == cl.ERR_NONFINITE


@pytest.mark.parametrize("layer", [0, 8, 9])
@pytest.mark.parametrize("fmt", FORMATS)
def test_full_size_sdxl_projection_inputs(cl, layer, fmt):
    """Full-size activations of the SDXL projection workload (bucket 9, heaviest tails)."""
    X = WL.sdxl_layer_activation(layer, 9)
    compare(cl, X, fmt)

"""GPU exhaustive activation-format argmin (Eq. format-argmin) against the oracle: the five
squared-error sums within 1e-5 relative (fp32 element errors, fp64 sums), the argmin equal
except at near-ties, exact zeros where a format reproduces the tensor."""
import numpy as np
import pytest

from oracle import select as SEL
from oracle import formats as F
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host

pytestmark = pytest.mark.gpu
RTOL = 1e-5


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def gpu_sse(cl, X):
    import torch
    out, st = cl.act_format_sse(cuda(X))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return host(out)


def check(cl, X, what):
    got = gpu_sse(cl, X)
    ref = SEL.act_format_sse(X)
    np.testing.assert_allclose(got, ref, rtol=RTOL, atol=1e-30, err_msg=what)
    f_ref = SEL.act_format_argmin(ref)
    f_got = cl.act_format_argmin(got)
    if f_got != f_ref:   # only where the two best errors are within the tolerance of each other
        assert abs(ref[f_got] - ref[f_ref]) <= 2 * RTOL * ref[f_ref], what
    return got


@pytest.mark.parametrize("shape", [(1, 32), (3, 64), (257, 96), (1000, 4096)])
@pytest.mark.parametrize("nu", [3, 5, 30])
def test_ragged_shapes_and_tails(cl, shape, nu):
    g = np.random.default_rng(shape[0] * 31 + nu)
    X = WL.to_fp16(g.standard_t(nu, shape) * 2.0 ** g.integers(-8, 6))
    check(cl, X, "%s nu %d" % (shape, nu))


def test_exact_format_gives_zero(cl):
    """E4M3 grid values with 448 in every 32-element block: per-tensor E4M3 (s = 1) and MXFP8
    (every block exponent 0) are exact on the GPU too."""
    vals = np.array([float(v) for v in F.fp_decode(np.arange(0x08, 0x7F), "e4m3")])
    g = np.random.default_rng(5)
    x = g.choice(vals, (64, 128)) * g.choice([-1.0, 1.0], (64, 128))
    x[:, ::32] = 448.0
    X = x.astype(np.float16)
    got = gpu_sse(cl, X)
    assert got[F.A_E4M3] == 0 and got[F.A_MXFP8] == 0 and got[F.A_INT8_ASYM] > 0
    assert cl.act_format_argmin(got) == F.A_E4M3


def test_calls_accumulate(cl):
    import torch
    g = np.random.default_rng(8)
    A, B = (WL.to_fp16(g.standard_t(4, (128, 256))) for _ in range(2))
    out, st = cl.act_format_sse(cuda(A))
    cl.act_format_sse(cuda(B), out=out, dev_status=st)
    torch.cuda.synchronize()
    np.testing.assert_allclose(host(out), SEL.act_format_sse(A) + SEL.act_format_sse(B), rtol=RTOL)


def test_nonfinite_input_sets_status(cl):
    import torch
    X = WL.to_fp16(np.random.default_rng(1).standard_normal((64, 256)))
    X[5, 9] = np.float16(np.inf)
    _, st = cl.act_format_sse(cuda(X))
    torch.cuda.synchronize()
    assert int(st.item()) == cl.ERR_NONFINITE


@pytest.mark.parametrize("layer", [0, 4, 9])
@pytest.mark.parametrize("bucket", [0, 5, 9])
def test_full_size_sdxl_activations(cl, layer, bucket):
    """The benchmark's SDXL activations (8192 x 640, 2048 x 1280, 2048 x 5120) at three buckets."""
    X = WL.sdxl_layer_activation(layer, bucket)
    check(cl, X, "layer %d bucket %d" % (layer, bucket))

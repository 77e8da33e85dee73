"""GPU group-wise weight formats and the per-linear (g, f) search of the DiT and few-step forks
(Sec. 3.5) against the oracle: packed codes, zero points and fp16 group scales bit-exact, linear
outputs within 2^-10 sum|a w| of the fp64 product of the same dequantized operands (the GPU's
fp16 weight operand equals the oracle's DQ exactly), search scores within 1e-5 relative."""
import numpy as np
import pytest

import blob as B
from oracle import formats as F
from oracle import gemm as G
from oracle import select as SEL
from oracle.nf4 import nf4_levels_fp16
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host, assert_within_bound

pytestmark = pytest.mark.gpu
GROUPED = [F.W_INT8_SYM, F.W_INT8_ASYM, F.W_INT4_SYM, F.W_INT4_ASYM, F.W_NF4, F.W_E2M1]
RTOL = 1e-5


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def pack_grouped(cl, W, fmt, g):
    import torch
    N, K = W.shape
    d = cl.pack_plan_grouped(N, K, fmt, g)
    blob, st = cl.pack_weights(cuda(W), cuda(np.full(N, fmt, np.uint8)), d)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return d, blob


@pytest.mark.parametrize("fmt", GROUPED)
@pytest.mark.parametrize("g", [32, 64, 192, 288])
def test_packed_blob_matches_oracle(cl, fmt, g):
    """Codes, per-block zero points and fp16 group scales of every channel, bit for bit; K = 320
    leaves a short last group for g = 192 and 288 and a padded last K-chunk."""
    rng = np.random.default_rng(fmt * 10 + g)
    N, K = 130, 320
    W = WL.weight_mix(rng, N, K)
    d, blob = pack_grouped(cl, W, fmt, g)
    desc, chans = B.unpack(host(blob).tobytes())
    assert desc["group"] == g and desc["version"] == 3
    L = nf4_levels_fp16()
    q = F.weight_quant_grouped(W, fmt, g, nf4_levels=L)
    asym = fmt in (F.W_INT8_ASYM, F.W_INT4_ASYM)
    for c in range(N):
        ch = chans[c]
        assert ch["fmt"] == fmt and ch["s"] == np.float32(1.0)
        for k0, k1, qq in q["groups"]:
            np.testing.assert_array_equal(ch["codes"][k0:k1], qq["codes"][c], err_msg="channel %d" % c)
            blocks = slice(k0 // 32, k1 // 32)
            assert np.all(ch["gscale16"][blocks] == np.float16(qq["s"][c]))
            assert np.all(ch["e8m0"][blocks] == (qq["z"][c] if asym else 0))


@pytest.mark.parametrize("fmt", GROUPED)
@pytest.mark.parametrize("g", [32, 128, 288])
@pytest.mark.parametrize("act_fmt", [F.A_E4M3, F.A_INT8_ASYM, F.A_FP16])
def test_grouped_linear_matches_oracle(cl, fmt, g, act_fmt):
    import torch
    rng = np.random.default_rng(100 + fmt * 7 + g + act_fmt)
    M, K, N = 200, 320, 257
    X = WL.to_fp16(rng.standard_t(4, (M, K)))
    W = WL.weight_mix(rng, N, K)
    bias = rng.normal(0, 0.02, N).astype(np.float32)
    d, blob = pack_grouped(cl, W, fmt, g)
    Y, st = cl.linear(cuda(X), d, blob, act_fmt, bias=cuda(bias))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    L = nf4_levels_fp16()
    w = F.weight_dequant_grouped(F.weight_quant_grouped(W, fmt, g, nf4_levels=L), nf4_levels=L)
    a = X.astype(np.float64) if act_fmt == F.A_FP16 else F.act_dequant(F.act_quant(X, act_fmt))
    y_ref, bound = G.linear_rows_reference(a, w, np.arange(M), bias)
    assert_within_bound(host(Y), y_ref, bound, "fmt %d g %d act %d" % (fmt, g, act_fmt))


def test_channel_energy_matches_oracle(cl):
    import torch
    rng = np.random.default_rng(3)
    A = WL.to_fp16(rng.standard_t(4, (1000, 1152)))
    Bm = WL.to_fp16(rng.standard_normal((37, 1152)) * 3)
    e = cl.act_channel_energy(cuda(A))
    cl.act_channel_energy(cuda(Bm), energy=e)
    torch.cuda.synchronize()
    np.testing.assert_allclose(host(e), SEL.input_energy(A) + SEL.input_energy(Bm), rtol=1e-6)


def check_search(cl, W, pal, groups, energy=None, what=""):
    import torch
    mask = sum(1 << f for f in pal)
    scores = cl.select_weight_groups(cuda(W), mask, cl.group_mask(groups),
                                     energy=None if energy is None else cuda(energy))
    torch.cuda.synchronize()
    got = host(scores)
    (gb, fb), ref, cands = SEL.select_grouped(W, pal, groups, energy=energy)
    assert cl.group_candidates(mask, cl.group_mask(groups)) == cands
    np.testing.assert_allclose(got, ref, rtol=RTOL, err_msg=what)
    i = cl.candidate_argmin(got)
    j = cands.index((gb, fb))
    if i != j:  # only at a near-tie
        assert abs(ref[i] - ref[j]) <= 2 * RTOL * ref[j], what
    return cands[i]


@pytest.mark.parametrize("pal", [[F.W_INT4_ASYM, F.W_NF4, F.W_E2M1],
                                 [F.W_INT4_ASYM, F.W_NF4, F.W_E2M1, F.W_MXINT4, F.W_MXFP4],
                                 [F.W_INT8_SYM, F.W_INT8_ASYM, F.W_MXINT8]])
@pytest.mark.parametrize("shape", [(1, 32), (37, 320), (300, 1152)])
def test_search_scores_match_oracle(cl, pal, shape):
    rng = np.random.default_rng(shape[0] + len(pal))
    W = WL.weight_mix(rng, *shape)
    check_search(cl, W, pal, F.GROUP_SIZES, what="%s %s" % (pal, shape))


def test_input_aware_search_on_pixart_layer(cl):
    """A PixArt-alpha attention projection (K = N = 1152) with input-channel energies from seeded
    activations whose channels differ in scale (the DiT case the input-aware SQNR targets): GPU
    energies, GPU search, then the chosen (g, f) packed and multiplied, checked on 64 rows."""
    import torch
    rng = np.random.default_rng(11)
    M, K, N = 512, 1152, 1152
    X = WL.to_fp16(rng.standard_t(5, (M, K)) * np.exp(rng.normal(0, 1.0, K))[None, :])
    W = WL.weight_mix(rng, N, K)
    e_dev = cl.act_channel_energy(cuda(X))
    torch.cuda.synchronize()
    energy = host(e_dev)
    np.testing.assert_allclose(energy, SEL.input_energy(X), rtol=1e-6)
    g, f = check_search(cl, W, [F.W_INT4_ASYM, F.W_NF4, F.W_E2M1], F.GROUP_SIZES, energy=energy, what="pixart")
    d, blob = pack_grouped(cl, W, f, g)
    Y, st = cl.linear(cuda(X), d, blob, F.A_E5M2)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    L = nf4_levels_fp16()
    w = F.weight_dequant_grouped(F.weight_quant_grouped(W, f, g, nf4_levels=L), nf4_levels=L)
    rows = np.sort(rng.choice(M, 64, replace=False))
    a = F.act_dequant(F.act_quant(X, F.A_E5M2))
    y_ref, bound = G.linear_rows_reference(a, w, rows, None)
    assert_within_bound(host(Y)[rows], y_ref, bound, "pixart (g %d, f %d)" % (g, f))

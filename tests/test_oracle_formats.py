"""Pins of the oracle's number formats against what the paper fixes (App. A.11, App. A.7).

Each test checks the oracle against an independent construction: the grids against the
numbers printed in App. A.11, the rounding against a nearest-value search over a grid built
from the exponent/mantissa definition, the scale rules against their closed forms.
"""
import numpy as np
import pytest

from oracle import formats as F

RNG = np.random.default_rng(20260001)


def grid_from_definition(ebits, mbits, bias, nan_rule):
    """Positive finite values and their mantissa parity, enumerated from the bit definition."""
    vals, even = [], []
    for E in range(1 << ebits):
        for M in range(1 << mbits):
            if nan_rule(E, M):
                continue
            if E == 0:
                v = M / (1 << mbits) * 2.0 ** (1 - bias)
            else:
                v = (1 + M / (1 << mbits)) * 2.0 ** (E - bias)
            vals.append(v)
            even.append(M % 2 == 0)
    order = np.argsort(vals)
    return np.asarray(vals)[order], np.asarray(even)[order]


GRIDS = {
    "e4m3": grid_from_definition(4, 3, 7, lambda E, M: E == 15 and M == 7),
    "e5m2": grid_from_definition(5, 2, 15, lambda E, M: E == 31),
    "e2m1": grid_from_definition(2, 1, 1, lambda E, M: False),
}


def naive_round(v, name):
    """Nearest finite grid value by search; ties to the even mantissa; beyond the largest
    finite value -> the largest finite value (saturation)."""
    grid, even = GRIDS[name]
    a = np.abs(v)
    out = np.empty_like(a)
    hi_idx = np.clip(np.searchsorted(grid, a, side="left"), 0, len(grid) - 1)
    for i, (x, j) in enumerate(zip(a, hi_idx)):
        if x >= grid[-1]:
            out[i] = grid[-1]
            continue
        up = grid[j]
        lo_j = j - 1 if grid[j] > x else j
        lo = grid[max(lo_j, 0)]
        if up - x < x - lo:
            out[i] = up
        elif x - lo < up - x:
            out[i] = lo
        else:
            out[i] = up if even[j] else lo
    return np.copysign(out, v)


# ------------------------------------------------------------------ grids (App. A.11)
def test_e4m3_grid():
    codes = np.arange(256)
    v = F.fp_decode(codes, "e4m3")
    nan = np.isnan(v)
    assert list(codes[nan]) == [0x7F, 0xFF]                 # no infinities, one NaN per sign
    fin = v[~nan]
    assert fin.max() == 448.0 and fin.min() == -448.0       # App. A.11: E4M3 spans +-448
    pos = np.unique(fin[fin > 0])
    assert pos.min() == 2.0 ** -9                           # smallest subnormal m * 2^-9
    assert F.fp_decode(0x08, "e4m3") == 2.0 ** -6           # App. A.11: smallest normal 2^-6
    assert np.all(np.diff(pos[(pos >= 1) & (pos < 2)]) == 2.0 ** -3)   # 3 mantissa bits
    np.testing.assert_array_equal(pos, GRIDS["e4m3"][0][1:])


def test_e5m2_grid():
    v = F.fp_decode(np.arange(256), "e5m2")
    fin = v[np.isfinite(v)]
    assert fin.max() == 57344.0                             # App. A.11: E5M2 spans +-57344
    assert F.fp_decode(0x04, "e5m2") == 2.0 ** -14          # App. A.11: smallest normal 2^-14
    assert np.sum(~np.isfinite(v)) == 8                     # exponent 31: inf and NaN
    pos = np.unique(fin[fin > 0])
    assert np.all(np.diff(pos[(pos >= 1) & (pos < 2)]) == 2.0 ** -2)   # 2 mantissa bits


def test_e2m1_grid_matches_paper():
    v = F.fp_decode(np.arange(16), "e2m1")
    printed = {0, 0.5, 1, 1.5, 2, 3, 4, 6}                  # App. A.11, FP4 E2M1
    assert set(np.abs(v).tolist()) == printed
    assert sorted(v[:8].tolist()) == sorted(printed)
    assert np.all(v[8:] == -v[:8])


# ------------------------------------------------------------------ round trips
@pytest.mark.parametrize("name,ncodes", [("e4m3", 256), ("e5m2", 256), ("e2m1", 16)])
def test_code_round_trip(name, ncodes):
    codes = np.arange(ncodes)
    v = F.fp_decode(codes, name)
    ok = np.isfinite(v)
    np.testing.assert_array_equal(F.fp_quantize(v[ok], name), codes[ok])


@pytest.mark.parametrize("name", ["e4m3", "e5m2", "e2m1"])
def test_rounding_against_search(name):
    grid, _ = GRIDS[name]
    mids = (grid[:-1] + grid[1:]) / 2
    mids32 = mids.astype(np.float32)
    near = np.concatenate([mids32, np.nextafter(mids32, np.float32(np.inf)),
                           np.nextafter(mids32, np.float32(0))])
    lo_e = int(np.floor(np.log2(grid[1]))) - 3
    hi_e = int(np.ceil(np.log2(grid[-1]))) + 2
    rnd = (RNG.uniform(1, 2, 20000) * 2.0 ** RNG.integers(lo_e, hi_e, 20000)).astype(np.float32)
    special = np.array([0.0, grid[-1], grid[-1] * 1.01, grid[-1] * 1e3, 2.0 ** (lo_e - 20)],
                       dtype=np.float32)
    v = np.concatenate([near, rnd, special]).astype(np.float64)
    v = np.concatenate([v, -v])
    np.testing.assert_array_equal(F.fp_round(v, name), naive_round(v, name))


def test_negative_values_rounding_to_zero_keep_sign():
    c = F.fp_quantize(np.array([-0.0, -1e-30, 1e-30]), "e4m3")
    assert list(c) == [0x80, 0x80, 0x00]


def test_saturation_not_nan():
    """App. A.7 note (ii): clamp before the cast, never a NaN or Inf code."""
    big = np.array([448.0, 449.0, 464.0, 500.0, 1e6, 3e38])
    assert list(F.fp_quantize(big, "e4m3")) == [0x7E] * 6
    assert list(F.fp_quantize(-big * 200, "e5m2")) == [0xFB] * 6


# ------------------------------------------------------------------ ScaleZP closed forms (App. A.7)
def test_int8_asym_scale_zero_point():
    for _ in range(200):
        lo = -float(RNG.uniform(0.01, 10))
        hi = float(RNG.uniform(0.01, 10))
        x = np.array([[lo, hi] + list(RNG.uniform(lo, hi, 62))], dtype=np.float16)
        q = F.act_quant(x, F.A_INT8_ASYM)
        lo16, hi16 = float(x.min()), float(x.max())
        s_ref = (hi16 - lo16) / 255                           # s = (hi - lo) / 255
        assert abs(q["s"] - s_ref) <= 1e-6 * s_ref
        assert abs(q["z"] - (-lo16 / s_ref)) <= 0.5 + 1e-4   # z = round(-lo / s)
        assert q["codes"][0, np.argmin(x[0])] == 0            # lo -> code 0
        assert q["codes"][0, np.argmax(x[0])] >= 254          # hi -> top code (up to RNE)


@pytest.mark.parametrize("fmt,fmax,top", [(F.A_E4M3, 448.0, 0x7E), (F.A_E5M2, 57344.0, 0x7B)])
def test_fp8_scale(fmt, fmax, top):
    x = (RNG.standard_t(3, (16, 64)) * 0.5).astype(np.float16)
    q = F.act_quant(x, fmt)
    amax = float(np.abs(x.astype(np.float32)).max())
    assert q["s"] == np.float32(np.float32(amax) / np.float32(fmax))   # s = amax / Fmax
    assert q["z"] == 0
    i = np.unravel_index(np.argmax(np.abs(x.astype(np.float32))), x.shape)
    assert q["codes"][i] & 0x7F == top                                 # amax -> +-Fmax


def test_int8_asym_one_sided_ranges_include_zero():
    """R4: the range is widened to include 0, so a single-signed tensor keeps an exact zero:
    all positive -> z = 0, s = hi / 255; all negative -> z = 255, s = -lo / 255."""
    x = np.array([[1.0, 2.0, 3.0] + [1.5] * 29], np.float16)
    q = F.act_quant(x, F.A_INT8_ASYM)
    assert q["z"] == 0 and q["s"] == np.float32(np.float32(3.0) / np.float32(255.0))
    assert q["codes"][0, 2] == 255 and q["codes"][0, 0] == 85                 # 1.0 / (3/255) = 85
    q = F.act_quant(-x, F.A_INT8_ASYM)
    assert q["z"] == 255 and q["s"] == np.float32(np.float32(3.0) / np.float32(255.0))
    assert q["codes"][0, 2] == 0 and q["codes"][0, 0] == 170
    w = np.array([[0.5, 1.0, 2.0, 4.0] * 8], np.float16)                       # weight channel, INT4-asym
    qw = F.weight_quant(w, F.W_INT4_ASYM)
    assert qw["z"][0] == 0 and qw["s"][0] == np.float32(np.float32(4.0) / np.float32(15.0))


def test_fp8_round_trip_on_representable_values():
    """DQ(Q(x)) == x when x already lies on the E4M3 grid and amax = 448 (inv = 1)."""
    vals = F.fp_decode(np.arange(0x7F), "e4m3")
    x = np.concatenate([vals, -vals, [448.0]]).astype(np.float16).reshape(1, -1)
    x = np.pad(x, ((0, 0), (0, (-x.shape[1]) % 32)))
    q = F.act_quant(x, F.A_E4M3)
    assert q["s"] == 1.0
    np.testing.assert_array_equal(F.act_dequant(q), x.astype(np.float64))


# ------------------------------------------------------------------ MX (Sec. 3.6, App. A.11/A.12)
@pytest.mark.parametrize("fmt,off", [(F.A_MXFP8, 8), (F.A_MXINT8, 0)])
def test_mx_shared_exponent(fmt, off):
    x = (RNG.standard_t(3, (8, 256)) * 0.5).astype(np.float16)
    x[0, :32] = 0                                   # an all-zero block
    q = F.act_quant(x, fmt)
    xb = np.abs(x.astype(np.float64)).reshape(8, 8, 32).max(axis=2)
    e = np.floor(np.log2(np.where(xb > 0, xb, 1.0))).astype(int)
    expect = np.where(xb > 0, e - off + 127, 0)
    np.testing.assert_array_equal(q["e8m0"], expect)
    # elements normalised by the shared scale stay below 2^(off+1) (the paper's (-2, 2) for off 0)
    X = q["e8m0"].astype(int) - 127
    v = np.abs(x.astype(np.float64)).reshape(8, 8, 32) * 2.0 ** (-X[..., None])
    assert np.all(v[xb > 0] < 2.0 ** (off + 1))


def test_mx_round_trip_on_representable_values():
    """MXINT8: blocks whose elements are k * 2^(X-6) with the block max at 2^X round-trip."""
    R, K = 4, 64
    X = RNG.integers(-10, 10, (R, K // 32))
    k = RNG.integers(-127, 128, (R, K)).reshape(R, K // 32, 32)
    k[..., 0] = 64                                   # element 2^X fixes the shared exponent
    x = (k * 2.0 ** (X[..., None] - 6)).reshape(R, K).astype(np.float16)
    assert np.all(x.astype(np.float64) == (k * 2.0 ** (X[..., None] - 6)).reshape(R, K))
    q = F.act_quant(x, F.A_MXINT8)
    np.testing.assert_array_equal(q["e8m0"], X + 127)
    np.testing.assert_array_equal(F.act_dequant(q), x.astype(np.float64))


def test_mxfp8_dq_is_exact_in_fp16():
    """Exactness reading R13: DQ of an MX activation code from an fp16 tensor is an fp16 value."""
    x = np.concatenate([(RNG.standard_t(3, (64, 128)) * 2.0 ** RNG.integers(-20, 12, (64, 1))),
                        RNG.integers(-3, 4, (4, 128)) * 2.0 ** -24]).astype(np.float16)
    for fmt in (F.A_MXFP8, F.A_MXINT8):
        dq = F.act_dequant(F.act_quant(x, fmt))
        assert np.all(dq.astype(np.float16).astype(np.float64) == dq)


# ------------------------------------------------------------------ weight codecs
def test_weight_int_codes_in_range_and_exact_dq():
    W = (RNG.normal(0, 0.02, (64, 128))).astype(np.float16)
    for fmt, lo, hi in [(F.W_INT8_SYM, -127, 127), (F.W_INT8_ASYM, 0, 255),
                        (F.W_INT4_SYM, -7, 7), (F.W_INT4_ASYM, 0, 15)]:
        q = F.weight_quant(W, fmt)
        assert q["codes"].min() >= lo and q["codes"].max() <= hi
        dq = F.weight_dequant(q)
        w = W.astype(np.float64)
        # every element lands within half a step of its own value (no wrong sign or scale); the
        # slack covers the two roundings of R6 (fp32 inv and fp32 product), |q| * 2^-21 steps
        step = q["s"].astype(np.float64)[:, None]
        assert np.all(np.abs(dq - w) <= (0.5 + 255 * 2.0 ** -21) * step)


def test_weight_e2m1_grid_channel_is_exact():
    """A channel that is an E2M1 grid vector times 6/amax-consistent scale reconstructs exactly."""
    g = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6])
    w = (np.tile(np.concatenate([g, -g]), 2) * 2.0 ** -7).astype(np.float16).reshape(1, -1)
    q = F.weight_quant(w, F.W_E2M1)
    np.testing.assert_array_equal(F.weight_dequant(q), w.astype(np.float64))


# ---------------------------------------------------------------- static scales (Alg. 1 / Alg. 2)
@pytest.mark.parametrize("fmt", [F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2])
def test_static_range_equal_to_own_range_is_the_dynamic_path(fmt):
    """Alg. 2 with the calibration range equal to the tensor's own range reduces to Alg. 3."""
    X = (np.random.default_rng(7).standard_t(3, (64, 96)) * 0.7).astype(np.float16)
    x = X.astype(np.float32)
    dyn = F.act_quant(X, fmt)
    sta = F.act_quant(X, fmt, lo=x.min(), hi=x.max())
    assert np.array_equal(dyn["codes"], sta["codes"]) and dyn["s"] == sta["s"] and dyn["z"] == sta["z"]


def test_static_int8_asym_closed_form_and_clamping():
    """Range [-1, 1]: s = 2/255, inv = 127.5, z = RNE(127.5) = 128; 0.5 -> RNE(63.75) + 128 = 192;
    values beyond the calibration range clamp to codes 0 and 255."""
    s, inv, z = F.scale_zp(F.A_INT8_ASYM, -1.0, 1.0)
    assert s == np.float32(2.0 / 255.0) and inv == np.float32(127.5) and z == 128
    X = np.array([[0.5, -0.5, 3.0, -3.0, 0.0]], np.float16)
    q = F.act_quant(X, F.A_INT8_ASYM, lo=-1.0, hi=1.0)
    assert list(q["codes"][0]) == [192, 64, 255, 0, 128]


@pytest.mark.parametrize("fmt,fmax", [(F.A_E4M3, 448.0), (F.A_E5M2, 57344.0)])
def test_static_fp8_scale_and_saturation(fmt, fmax):
    """Range [-2, 1]: amax = 2, s = 2/Fmax, inv = Fmax/2; x = 1 lands on Fmax/2 exactly; x = 3
    is beyond the range and saturates to Fmax (never NaN, note (ii))."""
    s, inv, z = F.scale_zp(fmt, -2.0, 1.0)
    assert s == np.float32(2.0 / fmax) and inv == np.float32(fmax / 2.0) and z == 0
    name = "e4m3" if fmt == F.A_E4M3 else "e5m2"
    q = F.act_quant(np.array([[1.0, 3.0, -3.0]], np.float16), fmt, lo=-2.0, hi=1.0)
    vals = F.fp_decode(q["codes"][0], name)
    assert list(vals) == [fmax / 2.0, fmax, -fmax]


# ---------------------------------------------------------------- per-sample scales (Alg. 3 per sample)
@pytest.mark.parametrize("fmt", F.ACT_FORMATS)
def test_per_sample_with_one_group_is_the_per_tensor_path(fmt):
    X = (np.random.default_rng(8).standard_t(3, (48, 64)) * 0.7).astype(np.float16)
    (q,) = F.act_quant_per_sample(X, fmt, 1)
    ref = F.act_quant(X, fmt)
    assert np.array_equal(q["codes"], ref["codes"]) and q["s"] == ref["s"] and q["z"] == ref["z"]


@pytest.mark.parametrize("fmt", F.ACT_FORMATS)
@pytest.mark.parametrize("k", [-3, 2, 5])
def test_per_sample_power_of_two_equivariance(fmt, k):
    """A sample that is another sample times 2^k gets the same codes and a scale 2^k times as
    large (the zero point unchanged; MX: block exponents shifted by k), whatever the other
    samples hold -- a per-tensor scale would couple them."""
    g = np.random.default_rng(9 + k)
    Y = (g.standard_t(4, (16, 64)) * 0.5).astype(np.float16)
    other = (g.standard_normal((16, 64)) * 40.0).astype(np.float16)
    X = np.vstack([Y, (Y.astype(np.float64) * 2.0 ** k).astype(np.float16), other])
    qs = F.act_quant_per_sample(X, fmt, 3)
    assert np.array_equal(qs[0]["codes"], qs[1]["codes"])
    if fmt in (F.A_MXFP8, F.A_MXINT8):
        nz = Y.reshape(16, 2, 32).astype(np.float32).any(axis=2)
        d = qs[1]["e8m0"].astype(int) - qs[0]["e8m0"].astype(int)
        assert np.all(d[nz] == k)
    else:
        assert np.float32(qs[1]["s"]) == np.float32(np.float32(qs[0]["s"]) * np.float32(2.0 ** k))
        assert qs[1]["z"] == qs[0]["z"]
    np.testing.assert_array_equal(F.act_dequant_per_sample(qs)[16:32], F.act_dequant(qs[0]) * 2.0 ** k)


def test_per_sample_zero_sample_is_degenerate_and_isolated():
    """An all-zero sample takes the degenerate parameters (s = 1, z = 0, R7) and dequantizes to
    exactly zero; its neighbours keep the parameters of their own ranges."""
    X = np.zeros((12, 32), np.float16)
    X[:4] = 0.25
    X[:4, 0] = -0.75
    X[8:] = np.linspace(-2, 6, 4 * 32).reshape(4, 32)
    qs = F.act_quant_per_sample(X, F.A_INT8_ASYM, 3)
    assert qs[1]["s"] == np.float32(1.0) and qs[1]["z"] == 0 and not qs[1]["codes"].any()
    assert qs[0]["s"] == F.act_quant(X[:4], F.A_INT8_ASYM)["s"] == np.float32(1.0 / 255.0)
    assert qs[2]["s"] == np.float32(8.0 / 255.0)
    assert not F.act_dequant_per_sample(qs)[4:8].any()
    with pytest.raises(ValueError):
        F.act_quant_per_sample(X, F.A_E4M3, 5)

"""Pins of the oracle's weight-format selection (Sec. 3.4) and NF4 construction.

Brute force: a second, naive implementation of every weight codec (nearest code by search over
the code list) on tiny tensors must give the same SSE and the same argmin.  Constructed
channels pin the tie rule (palette order) and zero-error cases.
"""
import math
import os

import numpy as np
import pytest

from oracle import formats as F
from oracle import select as SEL
from oracle import nf4

RNG = np.random.default_rng(20260010)
E2M1_POS = [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]


def nearest(v, grid, tie_pick):
    """Nearest member of `grid` to v; equal distances resolved by tie_pick(candidates)."""
    d = [abs(v - g) for g in grid]
    m = min(d)
    cands = [g for g, dd in zip(grid, d) if dd == m]
    return cands[0] if len(cands) == 1 else tie_pick(cands)


def even_int(c):
    return [x for x in c if x % 2 == 0][0]


def naive_roundtrip(w, fmt, L16):
    """DQ(Q(w)) for one channel (float32 values), by search over each format's code values."""
    w = np.asarray(w, dtype=np.float32)
    f32 = np.float32
    amax = f32(np.abs(w).max())
    out = np.zeros(len(w))
    if fmt in (F.W_INT8_SYM, F.W_INT4_SYM):
        qm = 127 if fmt == F.W_INT8_SYM else 7
        s = f32(amax / f32(qm)) if amax else f32(1)
        inv = f32(f32(qm) / amax) if amax else f32(1)
        for i, x in enumerate(w):
            q = nearest(float(f32(x * inv)), range(-qm, qm + 1), even_int)
            out[i] = q * float(s)
    elif fmt in (F.W_INT8_ASYM, F.W_INT4_ASYM):
        lv = 255 if fmt == F.W_INT8_ASYM else 15
        lo, hi = f32(min(w.min(), 0)), f32(max(w.max(), 0))
        d = f32(hi - lo)
        s = f32(d / f32(lv)) if d else f32(1)
        inv = f32(f32(lv) / d) if d else f32(1)
        z = nearest(float(f32(-lo * inv)), range(0, lv + 1), even_int) if d else 0
        for i, x in enumerate(w):
            t = nearest(float(f32(x * inv)), range(-lv - 1, 2 * lv + 2), even_int)
            q = min(max(t + z, 0), lv)
            out[i] = (q - z) * float(s)
    elif fmt == F.W_E2M1:
        s = f32(amax / f32(6)) if amax else f32(1)
        inv = f32(f32(6) / amax) if amax else f32(1)
        grid = sorted(set([-g for g in E2M1_POS] + E2M1_POS))
        even_codes = {0.0, 1.0, 2.0, 4.0}            # mantissa bit 0 in E2M1

        def tie(c):
            return [x for x in c if abs(x) in even_codes][0]
        for i, x in enumerate(w):
            v = float(f32(x * inv))
            v = max(min(v, 6.0), -6.0)
            out[i] = nearest(v, grid, tie) * float(s)
    elif fmt == F.W_NF4:
        s = amax if amax else f32(1)
        for i, x in enumerate(w):
            v = float(f32(x / s))
            out[i] = nearest(v, list(L16), lambda c: min(c)) * float(s)
    else:
        body = {F.W_MXINT8: ("int", 127, 6, 0), F.W_MXINT4: ("int", 7, 2, 0),
                F.W_MXFP4: ("fp", None, None, 2)}[fmt]
        for b0 in range(0, len(w), 32):
            blk = w[b0:b0 + 32].astype(np.float64)
            a = np.abs(blk).max()
            if a == 0:
                continue
            X = math.frexp(a)[1] - 1 - body[3]
            for i, x in enumerate(blk):
                v = x * 2.0 ** -X
                if body[0] == "int":
                    q = nearest(v * 2 ** body[2], range(-body[1], body[1] + 1), even_int)
                    out[b0 + i] = q * 2.0 ** (X - body[2])
                else:
                    grid = sorted(set([-g for g in E2M1_POS] + E2M1_POS))
                    vv = max(min(v, 6.0), -6.0)
                    out[b0 + i] = nearest(vv, grid, lambda c: [y for y in c
                                          if abs(y) in {0.0, 1.0, 2.0, 4.0}][0]) * 2.0 ** X
    return out


@pytest.mark.parametrize("mask,name", [(0b111, "W8"), (0b111111000, "W4")])
def test_select_matches_brute_force(mask, name):
    L16 = nf4.nf4_levels_fp16()
    N, K = 12, 64
    W = np.concatenate([RNG.normal(0, 0.02, (4, K)), RNG.laplace(0, 0.02, (4, K)),
                        RNG.uniform(-0.05, 0.05, (4, K))]).astype(np.float16)
    W[3, 5] *= 20                                            # an outlier channel
    fmt, sse, pal = SEL.select_formats(W, mask)
    w64 = W.astype(np.float64)
    for c in range(N):
        errs = [((w64[c] - naive_roundtrip(W[c].astype(np.float32), f, L16)) ** 2).sum()
                for f in pal]
        np.testing.assert_allclose(sse[c], errs, rtol=1e-12, atol=1e-30)
        assert fmt[c] == pal[int(np.argmin(errs))]


def test_zero_error_cases_and_palette_tie_order():
    K = 64
    ints = RNG.integers(-7, 8, K)
    ints[0] = 7
    w_int = (ints * 2.0 ** -9).astype(np.float16)            # exactly INT4-sym representable
    g = RNG.choice(E2M1_POS, K) * RNG.choice([-1, 1], K)
    g[0] = 6.0
    w_fp4 = (g * 2.0 ** -8).astype(np.float16)               # exactly E2M1 representable
    w_zero = np.zeros(K, np.float16)
    W = np.stack([w_int, w_fp4, w_zero])
    fmt, sse, pal = SEL.select_formats(W, 0b111111000)
    assert sse[0, pal.index(F.W_INT4_SYM)] == 0
    assert fmt[0] == F.W_INT4_SYM                            # ties with others -> first in order
    assert sse[1, pal.index(F.W_E2M1)] == 0
    assert fmt[1] in (F.W_INT4_SYM, F.W_INT4_ASYM, F.W_NF4, F.W_E2M1)
    assert sse[1, pal.index(fmt[1])] == 0
    assert fmt[2] == F.W_INT4_SYM                            # all zero: first palette member
    fmt8, _, _ = SEL.select_formats(W, 0b111)
    assert fmt8[2] == F.W_INT8_SYM


def test_sqnr_argmax_equals_sse_argmin():
    """Eq. weight-argmax: argmax SQNR == argmin SSE (the numerator is fixed per channel)."""
    W = RNG.standard_t(4, (32, 64)).astype(np.float16) * np.float16(0.02)
    fmt, sse, pal = SEL.select_formats(W, 0b111111000)
    energy = (W.astype(np.float64) ** 2).mean(axis=1, keepdims=True)
    sqnr = 10 * np.log10(energy / (sse / W.shape[1]))
    assert np.all(np.asarray(pal)[np.argmax(sqnr, axis=1)] == fmt)


# ------------------------------------------------------------------ NF4 (App. A.11 citation)
def test_nf4_structure():
    L = nf4.nf4_levels_fp16()
    assert len(L) == 16 and np.all(np.diff(L) > 0)
    assert L[0] == -1.0 and L[-1] == 1.0
    assert np.sum(L == 0) == 1 and np.sum(L < 0) == 7 and np.sum(L > 0) == 8


def test_nf4_quantiles_by_bisection():
    """Re-derive the quantiles by bisection of Phi(x) = erfc(-x / sqrt 2) / 2."""
    def ppf(p):
        lo, hi = -10.0, 10.0
        for _ in range(200):
            mid = 0.5 * (lo + hi)
            if 0.5 * math.erfc(-mid / math.sqrt(2)) < p:
                lo = mid
            else:
                hi = mid
        return 0.5 * (lo + hi)
    d = nf4.NF4_DELTA
    pos = [ppf(d + i * (0.5 - d) / 8) for i in range(8)]
    neg = [-ppf(d + i * (0.5 - d) / 7) for i in range(7)]
    v = np.sort(np.array(pos + [0.0] + neg)) / max(pos)
    np.testing.assert_allclose(nf4.nf4_levels_exact(), v, atol=1e-12)
    assert np.all(v.astype(np.float16).astype(np.float64) == nf4.nf4_levels_fp16())


def test_nf4_levels_match_the_published_qlora_table():
    """The levels against the NF4 table that QLoRA publishes (Appendix E of Dettmers et al., 2023;
    the source App. A.11 cites for NF4), a fact from outside this construction: a wrong outermost
    probability (e.g. 1 - 1/32 alone), a wrong count of negative quantiles or a missing
    normalisation moves some level by 1e-3 or more.  The published values are float32 renderings,
    hence the 1e-6 tolerance."""
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "nf4_qlora_levels.txt")
    rows = [line.split() for line in open(path) if line.strip() and not line.startswith("#")]
    assert [int(r[0]) for r in rows] == list(range(16))
    published = np.array([float(r[1]) for r in rows])
    np.testing.assert_allclose(nf4.nf4_levels_exact(), published, rtol=0, atol=1e-6)
    # the frozen fp16 levels are those values rounded to fp16
    assert np.all(published.astype(np.float16).astype(np.float64) == nf4.nf4_levels_fp16())


def test_nf4_exact_midpoints_go_to_the_lower_level():
    """R9: the code is the number of midpoints strictly below w/s, so a weight exactly on a
    midpoint takes the lower level.  Nine of the fifteen midpoints are fp16 values: with a 1.0 in
    the row (s = amax = 1) those weights sit exactly on them."""
    L = nf4.nf4_levels_fp16()
    mids = (L[:-1] + L[1:]) / 2.0
    idx = [i for i in range(15) if float(np.float16(mids[i])) == mids[i]]
    assert len(idx) >= 5
    row = np.array([1.0] + [mids[i] for i in idx], np.float16)[None, :]
    q = F.weight_quant(row, F.W_NF4, nf4_levels=L)
    assert q["s"][0] == 1.0 and q["codes"][0, 0] == 15
    assert q["codes"][0, 1:].tolist() == idx
    nudged = np.nextafter(row.astype(np.float16), np.float16(2.0))     # one fp16 ulp above: upper level
    nudged[0, 0] = 1.0
    assert F.weight_quant(nudged, F.W_NF4, nf4_levels=L)["codes"][0, 1:].tolist() == [i + 1 for i in idx]


# ---------------------------------------------------------------- activation-format argmin (Eq. format-argmin)
def fp8_grid(ebits, mbits, bias, skip):
    """(value, mantissa-is-even) of every non-negative finite value, from the bit definition."""
    out = []
    for E in range(1 << ebits):
        for M in range(1 << mbits):
            if skip(E, M):
                continue
            v = (M / (1 << mbits)) * 2.0 ** (1 - bias) if E == 0 else (1 + M / (1 << mbits)) * 2.0 ** (E - bias)
            out.append((v, M % 2 == 0))
    return sorted(out)


E4M3 = fp8_grid(4, 3, 7, lambda E, M: E == 15 and M == 7)
E5M2 = fp8_grid(5, 2, 15, lambda E, M: E == 31)


def naive_fp8(v, grid):
    """Nearest grid value to v (ties to the even mantissa), saturating beyond the largest."""
    a = abs(v)
    if a >= grid[-1][0]:
        return math.copysign(grid[-1][0], v)
    vals = [g for g, _ in grid]
    r = nearest(a, vals, lambda c: [g for g, e in grid if g in c and e][0])
    return math.copysign(r, v)


def f32(v):
    return float(np.float32(v))


def naive_act_dq(X, fmt):
    """An independent restatement of the five activation codecs, element by element: ScaleZP of
    the tensor's range (App. A.7) with x/s as a rounded product by the reciprocal, nearest code by
    search, and the MX shared exponent from frexp (OCP rule, body emax 8 for E4M3, 0 for int8)."""
    x = np.asarray(X).astype(np.float64)
    out = np.zeros_like(x)
    if fmt in (F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2):
        lo, hi = float(x.min()), float(x.max())
        if fmt == F.A_INT8_ASYM:
            lo_, hi_ = min(lo, 0.0), max(hi, 0.0)
            d = f32(hi_ - lo_)
            s, inv = (1.0, 1.0) if d == 0 else (f32(d / 255), f32(255 / d))
            z = 0 if d == 0 else min(max(nearest(f32(-lo_ * inv), range(-1, 257), even_int), 0), 255)
            for i, v in np.ndenumerate(x):
                t = f32(v * inv)
                q = min(max(nearest(t, range(math.floor(t) - 1, math.floor(t) + 3), even_int) + z, 0), 255)
                out[i] = (q - z) * s
        else:
            fmax, grid = (448.0, E4M3) if fmt == F.A_E4M3 else (57344.0, E5M2)
            amax = max(abs(lo), abs(hi))
            s, inv = (1.0, 1.0) if amax == 0 else (f32(amax / fmax), f32(fmax / amax))
            for i, v in np.ndenumerate(x):
                out[i] = naive_fp8(f32(v * inv), grid) * s
        return out
    for r in range(x.shape[0]):
        for b0 in range(0, x.shape[1], 32):
            blk = x[r, b0:b0 + 32]
            amax = float(np.abs(blk).max())
            if amax == 0:
                continue
            e = math.frexp(amax)[1] - 1                    # floor(log2 amax)
            if fmt == F.A_MXFP8:
                X_ = e - 8
                out[r, b0:b0 + 32] = [naive_fp8(v * 2.0 ** -X_, E4M3) * 2.0 ** X_ for v in blk]
            else:
                X_ = e
                out[r, b0:b0 + 32] = [min(max(nearest(v * 2.0 ** -X_ * 64, range(-128, 129), even_int), -127), 127)
                                      * 2.0 ** -6 * 2.0 ** X_ for v in blk]
    return out


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_act_format_sse_against_naive_codecs(seed):
    g = np.random.default_rng(300 + seed)
    X = (g.standard_t(3 + seed, (3, 64)) * 2.0 ** (seed - 1)).astype(np.float16)
    x = X.astype(np.float64)
    sse = SEL.act_format_sse(X)
    naive = [((x - naive_act_dq(X, f)) ** 2).sum() for f in F.ACT_FORMATS]
    np.testing.assert_allclose(sse, naive, rtol=1e-12, atol=0)
    assert SEL.act_format_argmin(sse) == int(np.argmin(naive))


def test_act_format_sse_zero_on_the_e4m3_grid():
    """A tensor of E4M3 grid values with 448 in every 32-element block: per-tensor E4M3 reproduces
    it exactly (s = 1), and so does MXFP8 (every block's shared exponent is 0); INT8-asym and E5M2
    cannot.  The argmin is E4M3, the earlier of the two exact formats.  (A block whose largest
    value is 1.875 * 2^e would not be exact under MXFP8: the OCP exponent maps it to 480, which
    saturates to 448.)"""
    vals = np.array([g for g, _ in E4M3 if g >= 2.0 ** -6], np.float64)
    g = np.random.default_rng(5)
    x = g.choice(vals, (4, 96)) * g.choice([-1.0, 1.0], (4, 96))
    x[:, ::32] = 448.0
    X = x.astype(np.float16)
    assert np.array_equal(X.astype(np.float64), x)
    sse = SEL.act_format_sse(X)
    assert sse[F.A_E4M3] == 0 and sse[F.A_MXFP8] == 0
    assert sse[F.A_INT8_ASYM] > 0 and sse[F.A_E5M2] > 0
    assert SEL.act_format_argmin(sse) == F.A_E4M3


@pytest.mark.parametrize("k", [-2, 3])
def test_act_format_sse_power_of_two_scaling(k):
    """Scaling X by 2^k scales every format's error by exactly 4^k (all five scale rules are
    power-of-two equivariant away from fp16 subnormals), so the argmin does not move."""
    X = (np.random.default_rng(6).standard_t(4, (8, 64)) * 4.0).astype(np.float16)
    X2 = (X.astype(np.float64) * 2.0 ** k).astype(np.float16)
    assert np.array_equal(X2.astype(np.float64), X.astype(np.float64) * 2.0 ** k)
    a, b = SEL.act_format_sse(X), SEL.act_format_sse(X2)
    np.testing.assert_array_equal(b, a * 4.0 ** k)
    assert SEL.act_format_argmin(a) == SEL.act_format_argmin(b)


def test_act_format_argmin_ties_and_zero_tensor():
    assert SEL.act_format_argmin([1.0, 1.0, 0.5, 0.5, 2.0]) == 2
    sse = SEL.act_format_sse(np.zeros((2, 32), np.float16))
    assert not sse.any() and SEL.act_format_argmin(sse) == 0


# ---------------------------------------------------------------- group-wise formats and the (g, f) search
GROUPED_W4 = [F.W_INT4_ASYM, F.W_NF4, F.W_E2M1]


def test_group_bounds_ragged_tail():
    assert F.group_bounds(320, 192) == [(0, 192), (192, 320)]
    assert F.group_bounds(320, 288) == [(0, 288), (288, 320)]
    assert F.group_bounds(1152, 288) == [(0, 288), (288, 576), (576, 864), (864, 1152)]
    assert F.group_bounds(64, 128) == [(0, 64)]


@pytest.mark.parametrize("fmt", [F.W_INT8_SYM, F.W_INT8_ASYM, F.W_INT4_SYM, F.W_INT4_ASYM, F.W_NF4, F.W_E2M1])
def test_one_group_is_the_per_channel_code(fmt):
    """A group as long as the row has the per-channel format's codes, scale and zero point."""
    W = (RNG.standard_normal((5, 96)) * 0.05).astype(np.float16)
    L = nf4.nf4_levels_fp16()
    (k0, k1, q), = F.weight_quant_grouped(W, fmt, 128, nf4_levels=L)["groups"]
    ref = F.weight_quant(W, fmt, nf4_levels=L)
    assert (k0, k1) == (0, 96)
    assert np.array_equal(q["codes"], ref["codes"]) and np.array_equal(q["s"], ref["s"])
    assert np.array_equal(q["z"], ref["z"])


def naive_grouped_dq(W, fmt, g):
    """Independent restatement: per group, the scale rule of Sec. 3.2 / App. A.7 in fp32, nearest
    code by search, then value x fp16(scale) rounded to fp16."""
    L = [float(v) for v in nf4.nf4_levels_fp16()]
    e2m1 = sorted(set(E2M1_POS + [-v for v in E2M1_POS]))
    w = np.asarray(W).astype(np.float64)
    out = np.zeros_like(w)
    for c in range(w.shape[0]):
        for k0, k1 in F.group_bounds(w.shape[1], g):
            seg = w[c, k0:k1]
            amax = float(np.abs(seg).max())
            if fmt == F.W_INT4_ASYM:
                lo, hi = min(float(seg.min()), 0.0), max(float(seg.max()), 0.0)
                d = f32(hi - lo)
                s, inv = (1.0, 1.0) if d == 0 else (f32(d / 15), f32(15 / d))
                z = 0 if d == 0 else min(max(nearest(f32(-lo * inv), range(-1, 17), even_int), 0), 15)
                vals = [min(max(nearest(f32(v * inv), range(-40, 41), even_int) + z, 0), 15) - z for v in seg]
            elif fmt == F.W_E2M1:
                s, inv = (1.0, 1.0) if amax == 0 else (f32(amax / 6), f32(6 / amax))
                even = (0.0, 1.0, 2.0, 4.0, -1.0, -2.0, -4.0)     # the values with an even mantissa bit
                vals = [nearest(f32(v * inv), e2m1, lambda cc: [x for x in cc if x in even][0]) for v in seg]
            else:
                s = amax if amax != 0 else 1.0
                vals = [nearest(f32(v / s), L, lambda cc: min(cc)) for v in seg]
            s16 = float(np.float16(s))
            out[c, k0:k1] = [float(np.float16(v * s16)) for v in vals]
    return out


@pytest.mark.parametrize("fmt", GROUPED_W4)
@pytest.mark.parametrize("g", [32, 64, 192])
def test_grouped_dq_against_naive(fmt, g):
    W = (RNG.standard_t(4, (3, 320)) * 0.03).astype(np.float16)
    L = nf4.nf4_levels_fp16()
    dq = F.weight_dequant_grouped(F.weight_quant_grouped(W, fmt, g, nf4_levels=L), nf4_levels=L)
    np.testing.assert_array_equal(dq, naive_grouped_dq(W, fmt, g))


def test_grouped_search_finds_the_exact_grid():
    """Rows built on an INT4-asym grid per 64-channel group, with power-of-two scales that differ
    between groups: (64, INT4-asym) reproduces them exactly and wins; 128 and coarser mix two
    scales in one group and do not."""
    g = np.random.default_rng(12)
    N, K = 4, 256
    W = np.zeros((N, K))
    for c in range(N):
        for k0 in range(0, K, 64):
            s = 2.0 ** g.integers(-9, -4)
            q = g.integers(0, 16, 64)
            q[0], q[1] = 0, 15                      # the group's range spans the whole grid
            W[c, k0:k0 + 64] = (q - 5) * s          # zero point 5: lo = -5 s, hi = 10 s
    W16 = W.astype(np.float16)
    assert np.array_equal(W16.astype(np.float64), W)
    (gb, fb), scores, cands = SEL.select_grouped(W16, GROUPED_W4)
    assert (gb, fb) == (32, F.W_INT4_ASYM) or (gb, fb) == (64, F.W_INT4_ASYM)
    assert scores[cands.index((64, F.W_INT4_ASYM))] == 0
    assert scores[cands.index((128, F.W_INT4_ASYM))] > 0


def test_energy_weighting():
    W = (RNG.standard_normal((6, 128)) * 0.02).astype(np.float16)
    pal = [F.W_INT4_ASYM, F.W_NF4]
    _, plain, cands = SEL.select_grouped(W, pal)
    _, const, _ = SEL.select_grouped(W, pal, energy=np.full(128, 3.0))
    np.testing.assert_allclose(const, 3.0 * plain, rtol=1e-13)
    e = np.zeros(128)
    e[77] = 2.5
    _, one, _ = SEL.select_grouped(W, pal, energy=e)
    for i, (g, f) in enumerate(cands):
        err = W.astype(np.float64)[:, 77] - SEL.grouped_dequant(W, g, f)[:, 77]
        assert one[i] == pytest.approx(2.5 * (err ** 2).sum(), rel=1e-13)
    X = np.array([[1.0, -2.0], [3.0, 0.5]], np.float16)
    np.testing.assert_array_equal(SEL.input_energy(X), [10.0, 4.25])


def test_candidate_order():
    c = SEL.group_candidates([F.W_INT4_ASYM, F.W_NF4, F.W_E2M1, F.W_MXINT4, F.W_MXFP4])
    assert c[:5] == [(32, 4), (32, 5), (32, 6), (32, 7), (32, 8)]
    assert c[5:8] == [(64, 4), (64, 5), (64, 6)] and len(c) == 5 + 4 * 3
    assert SEL.group_candidates([F.W_INT8_SYM, F.W_INT8_ASYM, F.W_MXINT8], (32, 64)) == [
        (32, 0), (32, 1), (32, 2), (64, 0), (64, 1)]

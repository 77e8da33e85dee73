"""Pins of the oracle's weight-format selection (Sec. 3.4) and NF4 construction.

Brute force: a second, naive implementation of every weight codec (nearest code by search over
the code list) on tiny tensors must give the same SSE and the same argmin.  Constructed
channels pin the tie rule (palette order) and zero-error cases.
"""
import math

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

"""Per-output-channel weight-format selection (Sec. 3.4, Eq. weight-argmax).

Test infrastructure (see ``oracle/__init__``).

For each output channel c the row W[c, :] is round-tripped through every format of the palette
and the format with the highest SQNR = 10 log10(E[W_c^2] / E[(W_c - DQ(Q(W_c)))^2]) wins.  The
numerator is the same for every format of one channel, so the argmax of SQNR is the argmin of the
squared error; it is computed as SSE_f(c) = sum_k (w - DQ_f(Q_f(w)))^2 in fp64 from the fp16 w and
the exact DQ.  Ties go to the earlier format in palette order (strict '<'), the order of Sec. 3.2:
INT8-sym, INT8-asym, MXINT8 at 8 bits; INT4-sym, INT4-asym, NF4, E2M1, MXINT4, MXFP4 at 4 bits.
A channel whose error is zero under every format (e.g. all zeros) therefore takes the first
member of the palette.
"""
import numpy as np

from . import formats as F
from .nf4 import nf4_levels_fp16


def palette_from_mask(mask):
    """Palette members (weight-format codes, ascending = palette order) of a bit mask."""
    return [f for f in range(9) if (mask >> f) & 1]


def sse_all(W, palette):
    """SSE_f(c) for every channel c and palette member f: float64 array N x len(palette)."""
    w64 = np.asarray(W).astype(np.float64)
    L = nf4_levels_fp16()
    out = np.zeros((w64.shape[0], len(palette)))
    for j, f in enumerate(palette):
        dq = F.weight_dequant(F.weight_quant(W, f, nf4_levels=L), nf4_levels=L)
        out[:, j] = ((w64 - dq) ** 2).sum(axis=1)
    return out


def select_formats(W, mask):
    """fmt[c] = first argmin over the palette of SSE_f(c) (Eq. weight-argmax).  Returns
    (fmt uint8 [N], sse float64 N x P, palette list)."""
    palette = palette_from_mask(mask)
    sse = sse_all(W, palette)
    idx = np.argmin(sse, axis=1)        # numpy argmin returns the first minimum: palette order
    return np.asarray(palette, dtype=np.uint8)[idx], sse, palette


def near_tie(sse_row, rel=1e-6):
    """True when the two smallest errors of a channel are within `rel` relative of each other:
    the only channels where a different (equally good) choice is accepted."""
    s = np.sort(np.asarray(sse_row))
    if len(s) < 2:
        return False
    return (s[1] - s[0]) <= rel * max(s[1], 1e-300)


def quantize_selected(W, fmt):
    """Logical pack: each channel encoded in its own format.  Returns a list of per-channel dicts
    (codes int64 [K], s fp32, z int, e8m0 uint8 [K/32] or None) in original channel order."""
    W = np.asarray(W)
    L = nf4_levels_fp16()
    out = []
    for c in range(W.shape[0]):
        q = F.weight_quant(W[c:c + 1], int(fmt[c]), nf4_levels=L)
        out.append({"fmt": int(fmt[c]), "codes": q["codes"][0], "s": np.float32(q["s"][0]),
                    "z": int(q["z"][0]),
                    "e8m0": None if q["e8m0"] is None else q["e8m0"][0]})
    return out


def dequant_selected(W, fmt):
    """DQ(Q(W)) with each channel in its selected format, float64 N x K."""
    W = np.asarray(W)
    L = nf4_levels_fp16()
    out = np.zeros(W.shape, dtype=np.float64)
    for f in np.unique(fmt):
        rows = np.nonzero(fmt == f)[0]
        q = F.weight_quant(W[rows], int(f), nf4_levels=L)
        out[rows] = F.weight_dequant(q, nf4_levels=L)
    return out


# ---------------------------------------------------------------- activation-format argmin (Eq. format-argmin)
def act_format_sse(X):
    """Squared quantization error of one activation tensor X (fp16, M x K) under every activation
    format at its native granularity (Sec. 3.1 and 3.2: the per-tensor formats with the ScaleZP
    of X's own range, the MX formats per 32-element block): SSE_f = sum (x - DQ_f(Q_f(x)))^2 in
    fp64, f = 0..4 in palette order.  Summing it over the calibration tensors of one (layer,
    bucket) gives the objective of Eq. format-argmin times their element count."""
    x64 = np.asarray(X).astype(np.float64)
    return np.array([((x64 - F.act_dequant(F.act_quant(X, f))) ** 2).sum() for f in F.ACT_FORMATS])


def act_format_argmin(sse):
    """f* = the first format of the activation palette with the least accumulated error (ties go
    to the earlier format, as in the weight selection)."""
    sse = np.asarray(sse, dtype=np.float64)
    best = 0
    for f in range(1, len(sse)):
        if sse[f] < sse[best]:
            best = f
    return best


# ---------------------------------------------------------------- per-linear (g, f) search (Sec. 3.5 forks)
def input_energy(X):
    """Activation energy of each input channel, sum_m x[m, k]^2 in fp64 (the input-aware SQNR of
    the DiT fork weights channel k's error by E[x_k^2]; the sum over the calibration rows is that
    expectation times their number, which leaves the argmax unchanged)."""
    x = np.asarray(X).astype(np.float64)
    return (x * x).sum(axis=0)


def group_candidates(palette, groups=F.GROUP_SIZES):
    """The (g, f) tuples searched, in order (ties go to the earlier one): g-major; at every g the
    non-MX members of the palette in palette order, and at g = 32 the MX members too (their block
    is 32 whatever g is searched)."""
    out = []
    for g in groups:
        for f in palette:
            if not F.W_IS_MX[f] or g == 32:
                out.append((g, f))
    return out


def grouped_dequant(W, g, f):
    """DQ of W in format f at group size g (MX formats: their own 32-element blocks)."""
    L = nf4_levels_fp16()
    if F.W_IS_MX[f]:
        return F.weight_dequant(F.weight_quant(W, f))
    return F.weight_dequant_grouped(F.weight_quant_grouped(W, f, g, nf4_levels=L), nf4_levels=L)


def select_grouped(W, palette, groups=F.GROUP_SIZES, energy=None):
    """Per-linear (g, f) choice: the candidate with the highest SQNR, i.e. the least weighted
    squared error sum_{c,k} e_k (w - DQ(w))^2 (the signal term sum e_k w^2 is the same for every
    candidate); e_k = 1 without activation energies.  Returns ((g, f), scores fp64, candidates)."""
    w64 = np.asarray(W).astype(np.float64)
    e = np.ones(w64.shape[1]) if energy is None else np.asarray(energy, dtype=np.float64)
    cands = group_candidates(palette, groups)
    scores = np.array([(((w64 - grouped_dequant(W, g, f)) ** 2) * e[None, :]).sum() for g, f in cands])
    best = 0
    for i in range(1, len(cands)):
        if scores[i] < scores[best]:
            best = i
    return cands[best], scores, cands

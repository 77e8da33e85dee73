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

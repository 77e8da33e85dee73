"""fp64 reference of the format-adaptive quantized linear layer.

Test infrastructure (see ``oracle/__init__``).

The layer computes Y = DQ(Q_a(X)) . DQ(Q_w(W))^T + b (Sec. 3.6, Alg. 2 / Alg. 3 followed by the
layer's matmul): the activation tensor is quantized in the format the LUT picks for (layer,
bucket) with its own dynamic range (Alg. 3), every weight channel in its selected format
(Sec. 3.4).  The reference multiplies the exact dequantized operands in fp64 (a library matmul
serves as the step) and adds the bias.  The accepted error of an fp32-accumulating kernel is
|Y - Y_ref| <= 2^-10 * sum_k |a_k w_k| per element, with a, w the same dequantized operands.
"""
import numpy as np

from . import formats as F
from .select import dequant_selected

TOL_REL = 2.0 ** -10


def linear_reference(X, act_fmt, W, wfmt, bias=None, lo=None, hi=None):
    """Returns (Y_ref float64 M x N, bound float64 M x N, A_dq, W_dq).  With lo, hi given, X is
    quantized with the static ScaleZP of that calibration range (Alg. 2), else with its own range
    (Alg. 3)."""
    X = np.asarray(X)
    if act_fmt == F.A_FP16:
        a = X.astype(np.float64)                      # weight-only fork (Sec. 3.5, SDXL-Turbo)
    else:
        a = F.act_dequant(F.act_quant(X, act_fmt, lo, hi))
    w = dequant_selected(W, np.asarray(wfmt))
    y = linear_output(a, w, bias)
    bound = TOL_REL * (np.abs(a) @ np.abs(w).T)
    return y, bound, a, w


def linear_output(a_dq, w_dq, bias=None):
    """Y = A W^T (+ bias) in fp64 on the dequantized operands (Sec. 3.6)."""
    y = np.asarray(a_dq, dtype=np.float64) @ np.asarray(w_dq, dtype=np.float64).T
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return y


def linear_rows_reference(a_dq, w_dq, rows, bias=None):
    """Reference on a subset of output rows (for outputs too large to compute in full)."""
    a = a_dq[rows]
    y = a @ w_dq.T
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return y, TOL_REL * (np.abs(a) @ np.abs(w_dq).T)

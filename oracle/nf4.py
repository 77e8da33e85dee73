"""NormalFloat-4 levels (the NF4 code the paper cites in App. A.11: Dettmers et al., 2023, QLoRA).

Test infrastructure (see ``oracle/__init__``).

Construction, restated from the QLoRA description: NF4 is built from quantiles of a unit normal so
that it has an exact zero.  The positive half takes 8 quantiles Phi^-1(p) at 9 evenly spaced
probabilities p from delta down to 1/2 (the last one, Phi^-1(1/2) = 0, is dropped); the negative
half takes 7 quantiles -Phi^-1(p) at 8 evenly spaced probabilities from delta to 1/2 (again
dropping the zero); one zero is added; all 16 values are divided by the largest, Phi^-1(delta),
so they span [-1, 1].  The outermost probability delta is the mean of 1 - 1/(2*15) and
1 - 1/(2*16), the offsets of a 15- and a 16-level quantile grid.

The levels are then frozen as fp16 values (reading R9): the codec, the selector and the
GEMM all use the fp16-rounded levels, so an NF4 weight decodes exactly in fp16.

Pinned (tests): the structure (16 sorted values, exactly one zero, L0 = -1, L15 = 1, 7 negative and
8 positive), an independent bisection of the normal CDF, and the NF4 table QLoRA publishes
(Appendix E of Dettmers et al., 2023) to 1e-6.
"""
import numpy as np
from scipy.special import ndtri   # Phi^-1 in double precision (Cephes ndtri)

NF4_DELTA = 0.5 * ((1.0 - 1.0 / 30.0) + (1.0 - 1.0 / 32.0))


def nf4_levels_exact():
    """The 16 NF4 levels in float64, ascending."""
    pos = ndtri(np.linspace(NF4_DELTA, 0.5, 9)[:-1])          # 8 positive quantiles
    neg = -ndtri(np.linspace(NF4_DELTA, 0.5, 8)[:-1])         # 7 negative quantiles
    v = np.concatenate([pos, [0.0], neg])
    v = v / v.max()
    return np.sort(v)


def nf4_levels_fp16():
    """The levels frozen as fp16 (returned as float64 holding the fp16 values)."""
    return nf4_levels_exact().astype(np.float16).astype(np.float64)

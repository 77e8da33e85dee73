"""Noise schedule, bucket index, kurtosis and the routing rule.

Test infrastructure (see ``oracle/__init__``).  Passages followed:
  * alpha_bar_t = prod_{s<=t} (1 - beta_s) and SNR(t) = alpha_bar_t / (1 - alpha_bar_t) -- Sec. 2.1,
    Eq. (snr); schedule ranges in App. A.1;
  * bucket index b = min(floor(t / bucket_size), B - 1) -- Alg. 2 and Alg. 3;
  * bucket midpoint t_b = b T/B + T/(2B) -- Sec. 3.3 and Alg. 1;
  * kurtosis kappa = E[(x - mu)^4] / (E[(x - mu)^2])^2 (population, non-excess) -- App. A.2,
    Eq. (kurt), recovered in closed form from the power sums of Alg. 1 (Sec. 3.5);
  * routing rule -- Sec. 3.3 (shortcut -> MXFP8; kappa > 5 or SNR < 0.2 -> E5M2;
    kappa <= 3 and SNR > 2 -> INT8-asym; otherwise E4M3).

Readings of passages the paper leaves open: timesteps are integers 0..T-1 with alpha_bar_t including beta_t (R17);
the scaled-linear betas interpolate linearly in sqrt(beta) (Stable-Diffusion schedule named by
App. A.11 names it scaled-linear), the linear betas linearly in beta; kappa := 0 when the variance is 0.
"""
import numpy as np

from .formats import A_INT8_ASYM, A_E4M3, A_E5M2, A_MXFP8

T_DEFAULT = 1000
B_DEFAULT = 10
KAPPA_LOW, KAPPA_HIGH = 3.0, 5.0      # Sec. 3.3
TAU_LOW, TAU_HIGH = 0.2, 2.0          # Sec. 3.3


def betas_scaled_linear(T=T_DEFAULT, beta_start=0.00085, beta_end=0.012):
    """beta_i = (sqrt(beta_start) + i (sqrt(beta_end) - sqrt(beta_start)) / (T - 1))^2."""
    return np.linspace(np.sqrt(beta_start), np.sqrt(beta_end), T, dtype=np.float64) ** 2


def betas_linear(T=T_DEFAULT, beta_start=1e-4, beta_end=0.02):
    """beta_i = beta_start + i (beta_end - beta_start) / (T - 1)."""
    return np.linspace(beta_start, beta_end, T, dtype=np.float64)


def alpha_bar(betas):
    """alpha_bar_t = prod_{s <= t} (1 - beta_s) for t = 0..T-1 (Sec. 2.1)."""
    return np.cumprod(1.0 - np.asarray(betas, dtype=np.float64))


def snr(betas):
    """SNR(t) = alpha_bar_t / (1 - alpha_bar_t) for every t (Eq. snr)."""
    ab = alpha_bar(betas)
    return ab / (1.0 - ab)


def bucket(t, T=T_DEFAULT, B=B_DEFAULT):
    """b = min(floor(t / bucket_size), B - 1) with bucket_size = T / B (Alg. 2, Alg. 3)."""
    bucket_size = T / B
    return min(int(np.floor(t / bucket_size)), B - 1)


def bucket_midpoint(b, T=T_DEFAULT, B=B_DEFAULT):
    """t_b = b T/B + T/(2B) (Sec. 3.3, Alg. 1)."""
    return b * T / B + T / (2 * B)


def bucket_mean_snr(betas, B=B_DEFAULT):
    """Arithmetic mean of SNR(t) over the integer t of each bucket (the 'bucket mean SNR' column
    of Tab. lutstats)."""
    s = snr(betas)
    T = len(s)
    return np.array([s[[t for t in range(T) if bucket(t, T, B) == b]].mean() for b in range(B)])


def power_sums(x):
    """The Alg. 1 accumulator for one tensor: n, sum x, sum x^2, sum x^3, sum x^4, min, max
    (fp64)."""
    x = np.asarray(x, dtype=np.float64).ravel()
    return {"n": x.size, "s1": x.sum(), "s2": (x ** 2).sum(), "s3": (x ** 3).sum(),
            "s4": (x ** 4).sum(), "lo": x.min(), "hi": x.max()}


def merge_sums(a, b):
    """Power sums are additive (Sec. 3.5): the accumulator of the union of two tensors."""
    return {"n": a["n"] + b["n"], "s1": a["s1"] + b["s1"], "s2": a["s2"] + b["s2"],
            "s3": a["s3"] + b["s3"], "s4": a["s4"] + b["s4"],
            "lo": min(a["lo"], b["lo"]), "hi": max(a["hi"], b["hi"])}


def kurtosis_from_sums(n, s1, s2, s3, s4):
    """kappa = m4 / m2^2 with the central moments recovered from raw power sums:
    mu = S1/n, m2 = S2/n - mu^2, m4 = S4/n - 4 mu S3/n + 6 mu^2 S2/n - 3 mu^4 (App. A.2, Eq. kurt;
    Alg. 1 'recovered in closed form')."""
    mu = s1 / n
    m2 = s2 / n - mu * mu
    m4 = s4 / n - 4.0 * mu * s3 / n + 6.0 * mu * mu * s2 / n - 3.0 * mu ** 4
    if m2 <= 0:
        return 0.0
    return m4 / (m2 * m2)


def kurtosis(x):
    ps = power_sums(x)
    return kurtosis_from_sums(ps["n"], ps["s1"], ps["s2"], ps["s3"], ps["s4"])


def route(kappa, snr_b, is_shortcut=False):
    """The routing rule of Sec. 3.3, evaluated at SNR(t_b)."""
    if is_shortcut:
        return A_MXFP8
    if kappa > KAPPA_HIGH or snr_b < TAU_LOW:
        return A_E5M2
    if kappa <= KAPPA_LOW and snr_b > TAU_HIGH:
        return A_INT8_ASYM
    return A_E4M3


def build_lut(kappa, betas, shortcut=None, T=T_DEFAULT):
    """F[l, b] = Route(kappa[l, b], SNR(t_b), is_shortcut(l)) for an L x B kappa table (Alg. 1,
    final loop).  t_b is rounded down to an integer timestep (t_b = 100 b + 50 is already one)."""
    kappa = np.asarray(kappa, dtype=np.float64)
    L, B = kappa.shape
    s = snr(betas)
    shortcut = np.zeros(L, bool) if shortcut is None else np.asarray(shortcut, bool)
    F = np.zeros((L, B), dtype=np.uint8)
    for b in range(B):
        snr_b = s[int(bucket_midpoint(b, T, B))]
        for l in range(L):
            F[l, b] = route(kappa[l, b], snr_b, shortcut[l])
    return F

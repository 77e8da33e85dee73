"""Pins of the oracle's schedule, bucket, kurtosis and routing code.

SNR: the bucket means printed in Tab. lutstats (tests/golden/lutstats_snr.txt) and the ranges of
App. A.1.  Kurtosis: the exact values of two-point and three-point distributions and the
population values of Gaussian (3) and Laplace (6) samples.  Route: the thresholds of Sec. 3.3 at
their boundaries and the phase boundaries stated in App. A.10 / A.11.
"""
import os

import numpy as np
import pytest

from oracle import schedule as S
from oracle import formats as F

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "lutstats_snr.txt")


def load_golden():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        sched, b, val, dec, flag = line.split()
        rows.append((sched, int(b), float(val), int(dec), int(flag)))
    return rows


@pytest.mark.parametrize("sched", ["scaled_linear", "linear"])
def test_bucket_mean_snr_matches_table(sched):
    betas = S.betas_scaled_linear() if sched == "scaled_linear" else S.betas_linear()
    means = S.bucket_mean_snr(betas)
    rows = [r for r in load_golden() if r[0] == sched]
    assert len(rows) == 10
    for _, b, printed, dec, flag in rows:
        unit = 10.0 ** -dec
        tol = unit if flag else 0.5 * unit
        assert abs(means[b] - printed) <= tol + 1e-12, (sched, b, means[b], printed)


def test_snr_ranges_app_a1():
    """SDXL ~1e3 at t=0 to ~1e-2 at t=T; PixArt ~1e4 to ~1e-4; monotone decreasing."""
    sl = S.snr(S.betas_scaled_linear())
    li = S.snr(S.betas_linear())
    assert 500 < sl[0] < 5000 and 1e-3 < sl[-1] < 1e-1
    assert 5e3 < li[0] < 5e4 and 1e-5 < li[-1] < 1e-3
    assert np.all(np.diff(sl) < 0) and np.all(np.diff(li) < 0)
    # closed form at t = 0: alpha_bar_0 = 1 - beta_0
    assert sl[0] == pytest.approx((1 - 0.00085) / 0.00085, rel=1e-12)
    assert li[0] == pytest.approx((1 - 1e-4) / 1e-4, rel=1e-12)


def test_bucket_index():
    assert [S.bucket(t) for t in (0, 99, 100, 550, 999, 1000, 1200)] == [0, 0, 1, 5, 9, 9, 9]
    assert [S.bucket_midpoint(b) for b in (0, 5, 9)] == [50, 550, 950]


def test_phase_boundaries_from_snr_gates():
    """App. A.10: INT8 only in SDXL buckets 0-2 (SNR > 2); E5M2 forced from b = 6 on SDXL and
    from b = 4 on PixArt (SNR < 0.2).  Evaluated at the bucket midpoint (Sec. 3.3)."""
    for betas, int8_ok, phase1 in [(S.betas_scaled_linear(), [0, 1, 2], list(range(6, 10))),
                                   (S.betas_linear(), None, list(range(4, 10)))]:
        s = S.snr(betas)
        mid = np.array([s[int(S.bucket_midpoint(b))] for b in range(10)])
        assert list(np.nonzero(mid < S.TAU_LOW)[0]) == phase1
        if int8_ok is not None:
            assert list(np.nonzero(mid > S.TAU_HIGH)[0]) == int8_ok


def test_kurtosis_exact_small_sets():
    assert S.kurtosis(np.array([-1.0, 1.0])) == pytest.approx(1.0, abs=1e-15)
    assert S.kurtosis(np.array([-1.0, 0.0, 0.0, 1.0])) == pytest.approx(2.0, abs=1e-15)
    # shifted and scaled sets: the central moments must be recovered from raw power sums
    assert S.kurtosis(7.5 + 3.0 * np.array([-1.0, 0.0, 0.0, 1.0])) == pytest.approx(2.0, rel=1e-9)
    # Bernoulli(p) on {0, 1}: kappa = (1 - 3p + 3p^2) / (p (1 - p))
    x = np.array([1.0] * 3 + [0.0] * 7)
    p = 0.3
    assert S.kurtosis(x) == pytest.approx((1 - 3 * p + 3 * p * p) / (p * (1 - p)), rel=1e-12)
    assert S.kurtosis(np.ones(10)) == 0.0


@pytest.mark.slow
def test_kurtosis_gaussian_and_laplace():
    rng = np.random.default_rng(20260002)
    assert S.kurtosis(rng.standard_normal(10_000_000)) == pytest.approx(3.0, abs=0.01)
    assert S.kurtosis(rng.laplace(size=10_000_000)) == pytest.approx(6.0, abs=0.1)
    assert S.kurtosis(2.0 + 0.1 * rng.standard_normal(1_000_000)) == pytest.approx(3.0, abs=0.03)


@pytest.mark.slow
def test_kurtosis_student_t_closed_form():
    """Student-t with nu > 4 degrees of freedom has kurtosis 3 + 6 / (nu - 4): 4 at nu = 10, the
    heavy-tailed family the synthetic activations are drawn from.  Its eighth moment exists, so
    the sample kurtosis of 10^7 draws has a spread of about 0.01."""
    rng = np.random.default_rng(20260004)
    assert S.kurtosis(rng.standard_t(10, 10_000_000)) == pytest.approx(4.0, abs=0.1)
    assert S.kurtosis(-1.5 + 0.5 * rng.standard_t(12, 10_000_000)) == pytest.approx(3.75, abs=0.1)


def test_power_sums_merge():
    rng = np.random.default_rng(20260003)
    a, b = rng.standard_normal(1000), rng.standard_t(5, 777)
    m = S.merge_sums(S.power_sums(a), S.power_sums(b))
    whole = S.power_sums(np.concatenate([a, b]))
    for k in ("n", "lo", "hi"):
        assert m[k] == whole[k]
    for k in ("s1", "s2", "s3", "s4"):
        assert m[k] == pytest.approx(whole[k], rel=1e-12, abs=1e-9)


def test_route_truth_table():
    eps = 1e-9
    assert S.route(100.0, 1e-9, True) == F.A_MXFP8                 # shortcut pin first
    assert S.route(5.0, 1.0) == F.A_E4M3                            # kappa > 5 is strict
    assert S.route(5.0 + eps, 1.0) == F.A_E5M2
    assert S.route(3.0, 0.2) == F.A_E4M3                            # SNR < 0.2 is strict
    assert S.route(3.0, 0.2 - eps) == F.A_E5M2
    assert S.route(3.0, 2.0) == F.A_E4M3                            # SNR > 2 is strict
    assert S.route(3.0, 2.0 + eps) == F.A_INT8_ASYM                 # kappa <= 3 inclusive
    assert S.route(3.0 + eps, 100.0) == F.A_E4M3
    assert S.route(2.0, 0.1) == F.A_E5M2                            # SNR gate overrides kappa


def test_lut_never_emits_mxint8():
    rng = np.random.default_rng(5)
    kappa = rng.uniform(1, 10, (50, 10))
    F_ = S.build_lut(kappa, S.betas_scaled_linear(), shortcut=rng.random(50) < 0.1)
    assert F.A_MXINT8 not in set(F_.ravel().tolist())       # Sec. 3.2: never emitted by Route

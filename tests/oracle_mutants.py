"""Plausible mistakes planted in the oracle, one at a time, to show that its pins catch them.

A pytest plugin (``-p oracle_mutants``) used by tests/test_oracle_mutants.py: when the environment
variable ORACLE_MUTANT names one of the mutants below, that mistake replaces the oracle function
for the whole run (the module attribute is swapped, so every caller sees it).  Each mutant is one
small slip of the kind that survives code review: a dropped term, a wrong sign, index, bound or
rounding rule, a transposed operand.  The oracle itself is never edited; nothing here runs unless
the variable is set.
"""
import os

import numpy as np


MUTANTS = (
    # number formats and scales
    "fp_round_ties_away", "fp_round_no_saturation", "fp_round_no_subnormal_floor",
    "e5m2_decode_inf_as_nan_only_for_max", "asym_zero_point_sign", "asym_raw_range",
    "fp8_amax_from_hi_only", "mxfp8_exponent_off_by_one", "mxint_exponent_off_by_one",
    "mx_zero_block_byte_127", "int8_sym_scale_over_128", "e2m1_weight_scale_over_4",
    "nf4_ties_to_upper_level", "nf4_delta_one_minus_1_32", "static_range_ignored", "per_sample_strided_rows",
    # schedule, statistics and route
    "kurtosis_dropped_term", "alpha_bar_excludes_t", "route_kappa_high_inclusive", "bucket_rounds_to_nearest",
    # selection and search
    "select_argmax", "select_abs_error", "act_argmin_last_tie", "act_sse_abs_error", "energy_abs",
    "candidates_mx_at_every_g", "group_tail_dropped", "grouped_scale_kept_in_fp32", "grouped_scores_unweighted",
    # the GEMM reference
    "gemm_weights_not_transposed", "gemm_bias_dropped",
)


def _fp_round_variant(F, ties_away=False, saturate=True, floor_binade=True):
    def fp_round(v, name):
        ebits, mbits, bias, vmax = F.FP_SPECS[name]
        v = np.asarray(v, dtype=np.float64)
        a = np.abs(v)
        emin = 1 - bias
        _, ex = np.frexp(a)
        e = np.maximum(ex - 1, emin) if floor_binade else ex - 1
        quantum = np.ldexp(1.0, e - mbits)
        r = (np.floor(a / quantum + 0.5) if ties_away else np.rint(a / quantum)) * quantum
        if saturate:
            r = np.minimum(r, vmax)
        return np.copysign(r, v)
    return fp_round


def _scale_zp_asym_variant(F, zero_sign=False, raw_range=False):
    def scale_zp_asym(lo, hi, levels):
        lo, hi = np.float32(lo), np.float32(hi)
        if not raw_range:
            lo = np.float32(min(lo, np.float32(0.0)))
            hi = np.float32(max(hi, np.float32(0.0)))
        d = np.float32(hi - lo)
        if d == 0:
            return np.float32(1.0), np.float32(1.0), 0
        s = np.float32(d / np.float32(levels))
        inv = np.float32(np.float32(levels) / d)
        z = int(F.rne(np.float32((lo if zero_sign else -lo) * inv)))
        return s, inv, min(max(z, 0), levels)
    return scale_zp_asym


def _kurtosis_without_cross_term(n, s1, s2, s3, s4):
    mu = s1 / n
    m2 = s2 / n - mu * mu
    m4 = s4 / n - 4.0 * mu * s3 / n - 3.0 * mu ** 4          # the 6 mu^2 S2 / n term dropped
    return 0.0 if m2 <= 0 else m4 / (m2 * m2)


def apply(name):
    from oracle import formats as F
    from oracle import gemm as G
    from oracle import schedule as S
    from oracle import select as SEL

    if name == "fp_round_ties_away":
        F.fp_round = _fp_round_variant(F, ties_away=True)
    elif name == "fp_round_no_saturation":
        F.fp_round = _fp_round_variant(F, saturate=False)
    elif name == "fp_round_no_subnormal_floor":
        F.fp_round = _fp_round_variant(F, floor_binade=False)
    elif name == "asym_zero_point_sign":
        F.scale_zp_asym = _scale_zp_asym_variant(F, zero_sign=True)
    elif name == "asym_raw_range":
        F.scale_zp_asym = _scale_zp_asym_variant(F, raw_range=True)
    elif name == "fp8_amax_from_hi_only":
        orig = F.scale_zp

        def scale_zp(fmt, lo, hi):
            if fmt in (F.A_E4M3, F.A_E5M2):
                s, inv = F.scale_sym(abs(np.float32(hi)), 448.0 if fmt == F.A_E4M3 else 57344.0)
                return s, inv, 0
            return orig(fmt, lo, hi)
        F.scale_zp = scale_zp
    elif name == "mxfp8_exponent_off_by_one":
        F.MX_BODIES["e4m3"] = 7
    elif name == "mxint_exponent_off_by_one":
        F.MX_BODIES["int8"] = 1
        F.MX_BODIES["int4"] = 1
    elif name == "nf4_ties_to_upper_level":
        orig = F.weight_quant

        def weight_quant(W, fmt, nf4_levels=None):
            q = orig(W, fmt, nf4_levels)
            if fmt == F.W_NF4:
                L = np.asarray(nf4_levels, dtype=np.float64)
                mids32 = ((L[:-1] + L[1:]) / 2.0).astype(np.float32)
                w = np.asarray(W).astype(np.float32)
                v = (w / q["s"][:, None]).astype(np.float32)
                q["codes"] = (mids32[None, None, :] <= v[..., None]).sum(axis=2).astype(np.int64)
            return q
        F.weight_quant = weight_quant
    elif name == "nf4_delta_one_minus_1_32":
        from oracle import nf4 as N
        N.NF4_DELTA = 1.0 - 1.0 / 32.0      # the 16-level offset alone instead of the mean of the two
    elif name == "kurtosis_dropped_term":
        S.kurtosis_from_sums = _kurtosis_without_cross_term
    elif name == "alpha_bar_excludes_t":
        S.alpha_bar = lambda betas: np.concatenate([[1.0], np.cumprod(1.0 - np.asarray(betas, np.float64))[:-1]])
    elif name == "route_kappa_high_inclusive":
        orig = S.route

        def route(kappa, snr_b, is_shortcut=False):
            if not is_shortcut and kappa == S.KAPPA_HIGH:
                return F.A_E5M2
            return orig(kappa, snr_b, is_shortcut)
        S.route = route
    elif name == "bucket_rounds_to_nearest":
        S.bucket = lambda t, T=S.T_DEFAULT, B=S.B_DEFAULT: min(int(np.rint(t / (T / B))), B - 1)
    elif name == "select_argmax":
        orig = SEL.select_formats

        def select_formats(W, mask):
            fmt, sse, palette = orig(W, mask)
            return np.asarray(palette, dtype=np.uint8)[np.argmax(sse, axis=1)], sse, palette
        SEL.select_formats = select_formats
    elif name == "select_abs_error":
        def sse_all(W, palette):
            w64 = np.asarray(W).astype(np.float64)
            L = SEL.nf4_levels_fp16()
            out = np.zeros((w64.shape[0], len(palette)))
            for j, f in enumerate(palette):
                dq = F.weight_dequant(F.weight_quant(W, f, nf4_levels=L), nf4_levels=L)
                out[:, j] = np.abs(w64 - dq).sum(axis=1)
            return out
        SEL.sse_all = sse_all
    elif name == "act_argmin_last_tie":
        def act_format_argmin(sse):
            sse = np.asarray(sse, dtype=np.float64)
            best = 0
            for f in range(1, len(sse)):
                if sse[f] <= sse[best]:
                    best = f
            return best
        SEL.act_format_argmin = act_format_argmin
    elif name == "act_sse_abs_error":
        SEL.act_format_sse = lambda X: np.array(
            [np.abs(np.asarray(X).astype(np.float64) - F.act_dequant(F.act_quant(X, f))).sum() for f in F.ACT_FORMATS])
    elif name == "energy_abs":
        SEL.input_energy = lambda X: np.abs(np.asarray(X).astype(np.float64)).sum(axis=0)
    elif name == "candidates_mx_at_every_g":
        SEL.group_candidates = lambda palette, groups=F.GROUP_SIZES: [(g, f) for g in groups for f in palette]
    elif name == "group_tail_dropped":
        F.group_bounds = lambda K, g: [(k0, k0 + g) for k0 in range(0, K - g + 1, g)] or [(0, K)]
    elif name == "gemm_weights_not_transposed":
        def linear_output(a_dq, w_dq, bias=None):
            y = np.asarray(a_dq, dtype=np.float64) @ np.asarray(w_dq, dtype=np.float64)
            return y if bias is None else y + np.asarray(bias, dtype=np.float64)[None, :]
        G.linear_output = linear_output
    elif name == "gemm_bias_dropped":
        orig = G.linear_output
        G.linear_output = lambda a_dq, w_dq, bias=None: orig(a_dq, w_dq, None)
    elif name == "grouped_scale_kept_in_fp32":
        def weight_dequant_grouped(q, nf4_levels=None):
            N = q["groups"][0][2]["codes"].shape[0]
            out = np.zeros((N, q["groups"][-1][1]))
            for k0, k1, qq in q["groups"]:
                v = F.weight_dequant(dict(qq, s=np.ones_like(qq["s"])), nf4_levels)
                out[:, k0:k1] = v * qq["s"].astype(np.float64)[:, None]      # no fp16 scale, no rounding
            return out
        F.weight_dequant_grouped = weight_dequant_grouped
    elif name == "grouped_scores_unweighted":
        orig = SEL.select_grouped
        SEL.select_grouped = lambda W, palette, groups=F.GROUP_SIZES, energy=None: orig(W, palette, groups, None)
    elif name == "per_sample_strided_rows":
        def act_quant_per_sample(X, fmt, n_groups):
            X = np.asarray(X)
            if n_groups < 1 or X.shape[0] % n_groups:
                raise ValueError("n_groups must divide M")
            return [F.act_quant(X[g::n_groups], fmt) for g in range(n_groups)]
        F.act_quant_per_sample = act_quant_per_sample
    elif name == "static_range_ignored":
        orig = F.act_quant
        F.act_quant = lambda X, fmt, lo=None, hi=None: orig(X, fmt)
    elif name == "mx_zero_block_byte_127":
        orig = F.mx_quant_rows

        def mx_quant_rows(x, body):
            codes, byte = orig(x, body)
            xb = np.asarray(x, np.float32).reshape(byte.shape[0], byte.shape[1], F.MX_BLOCK)
            return codes, np.where(np.abs(xb).max(axis=2) == 0, 127, byte).astype(np.uint8)
        F.mx_quant_rows = mx_quant_rows
    elif name == "int8_sym_scale_over_128":
        orig = F.weight_quant

        def weight_quant(W, fmt, nf4_levels=None):
            q = orig(W, fmt, nf4_levels)
            if fmt == F.W_INT8_SYM:
                w = np.asarray(W).astype(np.float32)
                for c in range(w.shape[0]):
                    q["s"][c], inv = F.scale_sym(np.abs(w[c]).max(), 128)
                    q["codes"][c] = np.clip(F.rne((w[c] * inv).astype(np.float32)), -127, 127)
            return q
        F.weight_quant = weight_quant
    elif name == "e2m1_weight_scale_over_4":
        orig = F.weight_quant

        def weight_quant(W, fmt, nf4_levels=None):
            q = orig(W, fmt, nf4_levels)
            if fmt == F.W_E2M1:
                w = np.asarray(W).astype(np.float32)
                for c in range(w.shape[0]):
                    q["s"][c], inv = F.scale_sym(np.abs(w[c]).max(), 4.0)
                    q["codes"][c] = F.fp_quantize((w[c] * inv).astype(np.float32), "e2m1")
            return q
        F.weight_quant = weight_quant
    elif name == "e5m2_decode_inf_as_nan_only_for_max":
        orig = F.fp_decode

        def fp_decode(code, name):
            v = orig(code, name)
            if name == "e5m2":
                c = np.asarray(code, dtype=np.int64)
                v = np.where((c & 0x7F) == 0x7B, np.nan, v)                    # max finite read as NaN
            return v
        F.fp_decode = fp_decode
    elif name != "none":
        raise ValueError("unknown oracle mutant %r" % (name,))


def pytest_configure(config):
    name = os.environ.get("ORACLE_MUTANT")
    if name:
        apply(name)

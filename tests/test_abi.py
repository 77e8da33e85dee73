"""The C-ABI library builds, loads and exports every entry point include/chameleon.h declares; its
host-only helpers (no GPU needed) agree with the oracle.  No kernel is launched here."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from oracle import schedule as S
from oracle import formats as F
from oracle import select as SEL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "chameleon.h")
# Tests that hand host buffers to entry points that take device pointers: every such call must be
# rejected on the host, so no kernel ever sees them.  They run only where no GPU is present, so a
# regression in the host checks can never launch a kernel on host memory.
host_buffers_only = pytest.mark.skipif(os.path.exists("/dev/nvidiactl"),
                                       reason="host-buffer argument checks run on GPU-less hosts only")


@pytest.fixture(scope="module")
def cl():
    from paper_2609_33496_gb300 import build
    build.build()
    import paper_2609_33496_gb300 as P
    P.chameleon.lib()
    return P.chameleon


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(chameleon_\w+)\s*\(", text)))


def test_exports_every_declared_symbol(cl):
    names = declared_symbols()
    assert len(names) >= 16
    L = ctypes.CDLL(cl.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", cl.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\b(chameleon_\w+)\b", out))
    assert set(names) == exported
    assert set(cl.EXPORTS) == set(names)


def test_bucket_matches_alg2(cl):
    for t in [0, 1, 99, 100, 101, 549, 550, 999, 1000, 1500]:
        assert cl.bucket(t) == S.bucket(t)
    assert cl.bucket(-1) == -1 and cl.bucket(5, 0, 10) == -1


@pytest.mark.parametrize("sched,betas", [(0, S.betas_scaled_linear()), (1, S.betas_linear())])
def test_snr_matches_oracle(cl, sched, betas):
    np.testing.assert_allclose(cl.snr(sched), S.snr(betas), rtol=1e-10)


def test_route_and_kurtosis_match_oracle(cl):
    rng = np.random.default_rng(7)
    for kappa in [1.0, 3.0, 3.0000001, 4.0, 5.0, 5.0000001, 9.0]:
        for snr_b in [0.1, 0.2, 0.2000001, 1.0, 2.0, 2.0000001, 50.0]:
            for sc in (False, True):
                assert cl.route(kappa, snr_b, sc) == S.route(kappa, snr_b, sc)
    for x in [rng.standard_normal(1000), 3 + rng.laplace(size=999), np.ones(5)]:
        ps = S.power_sums(x)
        sums = [ps["n"], ps["s1"], ps["s2"], ps["s3"], ps["s4"]]
        assert cl.kurtosis(sums) == pytest.approx(S.kurtosis_from_sums(*sums), rel=1e-12, abs=1e-15)


def test_pack_plan_layout(cl):
    fmt = np.array([F.W_NF4] * 50 + [F.W_INT4_SYM] * 130 + [F.W_MXFP4] * 3 + [F.W_E2M1] * 7, np.uint8)
    d = cl.pack_plan(len(fmt), 320, fmt)
    assert (d.N, d.K, d.Kp, d.bits) == (190, 320, 320, 4)
    assert list(d.n_class) == [140, 50] and list(d.n_tiles) == [2, 1]
    offs = [d.off_codes, d.off_scale, d.off_zero, d.off_e8m0, d.off_fmt, d.off_perm, d.bytes]
    assert all(o % 256 == 0 for o in offs) and offs == sorted(offs)
    assert d.off_scale - d.off_codes >= 3 * 5 * 128 * 32


def test_pack_plan_palette_matches_format_plan(cl):
    """A one-class palette gives the layout the selected formats would give, whatever they are."""
    rng = np.random.default_rng(5)
    fields = lambda d: (d.N, d.K, d.Kp, d.bits, list(d.n_class), list(d.n_tiles), d.off_codes, d.off_scale,
                        d.off_zero, d.off_e8m0, d.off_fmt, d.off_perm, d.bytes)
    cases = [(cl.PALETTE_W8, [F.W_INT8_SYM, F.W_INT8_ASYM, F.W_MXINT8], 300, 320),
             ((1 << F.W_INT4_ASYM) | (1 << F.W_E2M1) | (1 << F.W_MXINT4) | (1 << F.W_MXFP4),
              [F.W_INT4_ASYM, F.W_E2M1, F.W_MXINT4, F.W_MXFP4], 129, 96),
             (1 << F.W_NF4, [F.W_NF4], 1, 32)]
    for mask, members, N, K in cases:
        dp = cl.pack_plan_palette(N, K, mask)
        for _ in range(3):
            fmt = np.asarray(members, np.uint8)[rng.integers(0, len(members), N)]
            assert fields(dp) == fields(cl.pack_plan(N, K, fmt))
        assert [dp.n_fmt[f] for f in members] == [-1] * len(members)
    with pytest.raises(cl.ChameleonError) as e:
        cl.pack_plan_palette(64, 64, cl.PALETTE_W4)                # NF4 with class-0 formats
    assert e.value.status == cl.ERR_UNSUPPORTED
    for bad in (0, 0x200, 0x009):                                  # empty, out of range, mixed widths
        with pytest.raises(cl.ChameleonError) as e:
            cl.pack_plan_palette(64, 64, bad)
        assert e.value.status == cl.ERR_INVALID_ARG


def test_host_validation_errors(cl):
    with pytest.raises(cl.ChameleonError) as e:
        cl.pack_plan(4, 320, np.array([0, 0, 3, 3], np.uint8))     # mixed bit widths
    assert e.value.status == cl.ERR_INVALID_ARG
    with pytest.raises(cl.ChameleonError):
        cl.pack_plan(2, 100, np.array([0, 0], np.uint8))           # K not a multiple of 32
    with pytest.raises(cl.ChameleonError):
        cl.act_quant_size(16, 48, 1)
    with pytest.raises(cl.ChameleonError):
        cl.act_quant_size(16, 64, 7)
    q, w = cl.act_quant_size(256, 320, 3)
    assert q >= 256 * 320 + 256 + 256 * 10 and w == 0


def test_scale_zp_host_matches_oracle_bit_for_bit(cl):
    """The host ScaleZP (the static path's parameters, Alg. 1 / Alg. 2) gives the oracle's fp32 s,
    1/s and z for random, tiny, one-sided, degenerate and fp16-extreme ranges."""
    rng = np.random.default_rng(11)
    ranges = [(0.0, 0.0), (-1.0, -1.0), (2.0, 2.0), (-65504.0, 65504.0), (-1e-7, 3e-8), (0.0, 6.0),
              (-6.0, 0.0), (-0.5, 0.5), (-1.0, 254.0), (-254.0, 1.0), (-1.0 / 255, 1.0)]
    for _ in range(300):
        lo, hi = np.sort(rng.standard_normal(2) * 10.0 ** rng.uniform(-4, 4, 2))
        ranges.append((float(np.float32(lo)), float(np.float32(hi))))
    for fmt in (F.A_INT8_ASYM, F.A_E4M3, F.A_E5M2):
        for lo, hi in ranges:
            p = cl.scale_zp(fmt, lo, hi)
            s, inv, z = F.scale_zp(fmt, lo, hi)
            assert (np.float32(p.s), np.float32(p.inv), p.z, p.fmt) == (s, inv, z, fmt), (fmt, lo, hi)


@host_buffers_only
def test_scale_zp_and_static_entry_points_reject_bad_arguments(cl):
    for fmt, lo, hi in [(3, -1.0, 1.0), (5, -1.0, 1.0), (-1, 0.0, 1.0), (0, 1.0, -1.0),
                        (1, float("nan"), 1.0), (2, 0.0, float("inf")), (0, -3e38, 3e38)]:
        with pytest.raises(cl.ChameleonError) as e:
            cl.scale_zp(fmt, lo, hi)
        assert e.value.status == cl.ERR_INVALID_ARG
    L = cl.lib()
    dp = ctypes.byref(cl.pack_plan(64, 64, np.zeros(64, np.uint8)))  # a 64-input layer for the prepare calls
    buf = ctypes.create_string_buffer(1 << 16)
    x = ctypes.cast(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16, ctypes.c_void_p)
    good = cl.scale_zp(F.A_INT8_ASYM, -1.0, 3.0)
    bad = [None, cl.QParams(good.s, good.z, good.inv, F.A_E4M3), cl.QParams(0.0, 0, 1.0, 0),
           cl.QParams(1.0, 256, 1.0, 0), cl.QParams(float("inf"), 0, 1.0, 0), cl.QParams(1.0, -1, 1.0, 0)]
    for p in bad:
        ref = None if p is None else ctypes.byref(p)
        assert L.chameleon_act_quant_static(x, 16, 64, F.A_INT8_ASYM, ref, x, 1 << 15, x, None) == cl.ERR_INVALID_ARG
        assert L.chameleon_linear_prepare_static(x, 16, dp, F.A_INT8_ASYM, ref, x, 1 << 15, x,
                                                 None) == cl.ERR_INVALID_ARG
    fp8 = cl.scale_zp(F.A_E4M3, -1.0, 3.0)
    fp8.z = 1
    assert L.chameleon_act_quant_static(x, 16, 64, F.A_E4M3, ctypes.byref(fp8), x, 1 << 15, x,
                                        None) == cl.ERR_INVALID_ARG
    assert L.chameleon_act_quant_static(x, 16, 48, F.A_INT8_ASYM, ctypes.byref(good), x, 1 << 15, x,
                                        None) == cl.ERR_INVALID_ARG      # K not a multiple of 32


@host_buffers_only
def test_groups_and_output_type_argument_checks(cl):
    """Per-sample groups must divide M and number 1..CHAM_MAX_GROUPS; y_type is one of three.
    Every rejection happens on the host, before any launch."""
    L = cl.lib()
    dp = ctypes.byref(cl.pack_plan(64, 64, np.zeros(64, np.uint8)))  # a 64-input layer for the prepare calls
    buf = ctypes.create_string_buffer(1 << 20)
    x = ctypes.cast(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16, ctypes.c_void_p)
    for M, n in [(64, 0), (64, 65), (64, 3), (60, -1), (128, 128)]:
        assert L.chameleon_linear_prepare_groups(x, M, dp, F.A_E4M3, n, x, 1 << 19, x, None) == cl.ERR_INVALID_ARG
    d = cl.pack_plan(64, 64, np.zeros(64, np.uint8))
    for n, yt in [(3, cl.Y_F32), (0, cl.Y_F16), (1, 3), (1, -1), (65, cl.Y_BF16)]:
        assert L.chameleon_linear_gemm_ex(x, 64, ctypes.byref(d), x, F.A_E4M3, n, None, x, yt, x, 1 << 19, x,
                                          None) == cl.ERR_INVALID_ARG
    assert cl.MAX_GROUPS == 64


def test_act_format_argmin_host_helper(cl):
    for sse in ([3.0, 2.0, 2.0, 5.0, 1.0], [0.0] * 5, [1.0, 0.5, 0.25, 0.25, 0.5], [7, 7, 7, 7, 6.999]):
        assert cl.act_format_argmin(sse) == SEL.act_format_argmin(sse)
    assert cl.lib().chameleon_act_format_argmin(None) == -1
    w = ctypes.c_size_t()
    assert cl.lib().chameleon_act_format_sse_workspace_size(16, 48, ctypes.byref(w)) == cl.ERR_INVALID_ARG
    assert cl.lib().chameleon_act_format_sse_workspace_size(16, 64, ctypes.byref(w)) == cl.OK and w.value >= 256


def test_group_candidates_match_oracle(cl):
    for pal, groups in [([F.W_INT4_ASYM, F.W_NF4, F.W_E2M1], F.GROUP_SIZES),
                        ([F.W_INT4_ASYM, F.W_NF4, F.W_E2M1, F.W_MXINT4, F.W_MXFP4], F.GROUP_SIZES),
                        ([F.W_INT8_SYM, F.W_INT8_ASYM, F.W_MXINT8], (32, 128)),
                        ([F.W_MXFP4], (64,))]:
        mask = sum(1 << f for f in pal)
        assert cl.group_candidates(mask, cl.group_mask(groups)) == SEL.group_candidates(pal, groups)
    assert cl.candidate_argmin([3.0, 1.0, 1.0, 2.0]) == 1
    assert cl.lib().chameleon_candidate_argmin(None, 3) == -1


def test_pack_plan_grouped_layout_and_checks(cl):
    d = cl.pack_plan_grouped(300, 320, F.W_INT4_ASYM, 192)
    assert (d.group, d.bits, list(d.n_class), d.n_fmt[F.W_INT4_ASYM], d.version) == (192, 4, [300, 0], 300, 3)
    assert d.off_gscale % 256 == 0 and d.off_gscale >= d.off_perm + 4 * 384
    assert d.bytes >= d.off_gscale + 3 * 5 * 128 * 4
    assert cl.pack_plan(300, 320, np.full(300, F.W_INT4_ASYM, np.uint8)).off_gscale == 0
    for fmt, g, K in [(F.W_MXFP4, 32, 320), (F.W_NF4, 48, 320), (F.W_NF4, 0, 320), (F.W_E2M1, 32, 32 * 257),
                      (9, 32, 320)]:
        with pytest.raises(cl.ChameleonError) as e:
            cl.pack_plan_grouped(64, K, fmt, g)
        assert e.value.status == cl.ERR_INVALID_ARG
    w = ctypes.c_size_t()
    L = cl.lib()
    assert L.chameleon_select_weight_groups_workspace_size(64, 320, 0x070, 0, ctypes.byref(w)) == cl.ERR_INVALID_ARG
    assert L.chameleon_select_weight_groups_workspace_size(64, 320, 0x1F8 | 0x1, 1, ctypes.byref(w)) == cl.ERR_INVALID_ARG
    assert L.chameleon_select_weight_groups_workspace_size(64, 32 * 257, 0x070, 1, ctypes.byref(w)) == cl.ERR_INVALID_ARG
    assert L.chameleon_select_weight_groups_workspace_size(64, 320, 0x070, 0x1F, ctypes.byref(w)) == cl.OK


@host_buffers_only
def test_select_pack_palette_argument_checks(cl):
    L = cl.lib()
    buf = ctypes.create_string_buffer(1 << 20)
    x = ctypes.cast(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16, ctypes.c_void_p)
    d8 = cl.pack_plan_palette(64, 320, cl.PALETTE_W8)
    two = cl.pack_plan(64, 320, np.array([F.W_INT4_SYM, F.W_NF4] * 32, np.uint8))
    grouped = cl.pack_plan_grouped(64, 320, F.W_INT4_ASYM, 64)
    for d, N, K, mask in [(d8, 64, 256, cl.PALETTE_W8), (d8, 32, 320, cl.PALETTE_W8), (two, 64, 320, cl.PALETTE_W4),
                          (grouped, 64, 320, 1 << F.W_INT4_ASYM), (d8, 64, 320, cl.PALETTE_W4), (d8, 64, 320, 0)]:
        assert L.chameleon_select_pack_palette(x, N, K, mask, ctypes.byref(d), x, x, 1 << 19, x,
                                               None) == cl.ERR_INVALID_ARG


def test_check_rejects_a_null_status_word(cl):
    assert cl.lib().chameleon_check(None, None) == cl.ERR_INVALID_ARG


def test_linear_workspace_includes_split_k_partials(cl):
    """The GEMM splits K when its 128-channel x token tiles are fewer than half the SMs and K has at
    least 8 chunks of 64; the workspace then adds k_split x M x Np fp32 partial sums.  Up to 16
    tokens the weight-streaming kernel runs instead and needs none.  Without a device the library
    assumes the 152 SMs of a GB300."""
    sms = 152

    def bn(M):
        return next(b for b in (16, 32, 64, 128) if M <= b) if M <= 128 else 192

    def expected_extra(M, N, K):
        if M <= 16:          # the weight-streaming kernel: no split, no partial sums
            return 0
        tiles = -(-N // 128) * -(-M // bn(M))
        nk = -(-K // 64)
        if tiles * 2 > sms or nk < 8:
            return 0
        ks = max(1, min(sms // tiles, nk // 2))
        return -(-(ks * M * 128 * -(-N // 128) * 4) // 256) * 256

    for M, K, N in [(16, 1280, 1280), (154, 2048, 1280), (240, 4096, 1152), (2, 320, 1280), (2048, 1280, 10240),
                    (8192, 640, 640), (1, 512, 128)]:
        d = cl.pack_plan(N, K, np.full(N, F.W_INT8_SYM, np.uint8))
        base = cl.linear_workspace_size(M, d, F.A_FP16)          # FP16: 256 bytes before any partials
        assert base - 256 == expected_extra(M, N, K), (M, K, N)
        q = cl.linear_workspace_size(M, d, F.A_E4M3)
        assert q - (base - 256) >= 2 * M * K                      # the fp16 operand precedes the partials


def test_version_and_status_names(cl):
    assert cl.version() == 3
    assert cl.status_string(cl.OK) and cl.status_string(cl.ERR_TIMEOUT) != cl.status_string(cl.OK)


@host_buffers_only
@pytest.mark.parametrize("bad", [0, -1, -32])
def test_empty_and_negative_sizes_are_rejected_on_the_host(cl, bad):
    """Every entry point that takes a size rejects an empty (0) or negative M, N, K or count with
    CHAM_ERR_INVALID_ARG before touching the device (no GPU is present here)."""
    L = cl.lib()
    dp = ctypes.byref(cl.pack_plan(64, 64, np.zeros(64, np.uint8)))  # a 64-input layer for the prepare calls
    buf = ctypes.create_string_buffer(1 << 16)
    x = ctypes.cast(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16, ctypes.c_void_p)
    n = ctypes.c_size_t(0)
    d = cl.WPackDesc()
    good = cl.pack_plan(64, 64, np.zeros(64, np.uint8))
    p = cl.scale_zp(F.A_E4M3, -1.0, 1.0)
    calls = {
        "act_moments": lambda: L.chameleon_act_moments(x, bad, x, x, 1 << 15, None),
        "act_quant_size": lambda: L.chameleon_act_quant_size(bad, 64, 1, ctypes.byref(n), ctypes.byref(n)),
        "act_quant_size K": lambda: L.chameleon_act_quant_size(16, bad, 1, ctypes.byref(n), ctypes.byref(n)),
        "act_quant": lambda: L.chameleon_act_quant(x, bad, 64, 1, x, 1 << 15, x, 1 << 15, x, None),
        "act_quant K": lambda: L.chameleon_act_quant(x, 16, bad, 1, x, 1 << 15, x, 1 << 15, x, None),
        "act_quant_noalloc": lambda: L.chameleon_act_quant_noalloc(x, bad, 64, 1, x, 1 << 15, x, None),
        "act_quant_static": lambda: L.chameleon_act_quant_static(x, bad, 64, 1, ctypes.byref(p), x, 1 << 15, x,
                                                                 None),
        "act_format_sse_workspace_size": lambda: L.chameleon_act_format_sse_workspace_size(bad, 64,
                                                                                            ctypes.byref(n)),
        "act_format_sse": lambda: L.chameleon_act_format_sse(x, 16, bad, x, x, 1 << 15, x, None),
        "act_channel_energy": lambda: L.chameleon_act_channel_energy(x, bad, 64, x, None),
        "select_weight_formats": lambda: L.chameleon_select_weight_formats(x, bad, 64, cl.PALETTE_W8, x, None,
                                                                           None),
        "select_weight_formats K": lambda: L.chameleon_select_weight_formats(x, 16, bad, cl.PALETTE_W8, x,
                                                                             None, None),
        "select_weight_groups_workspace_size": lambda: L.chameleon_select_weight_groups_workspace_size(
            bad, 64, 1 << F.W_NF4, 1, ctypes.byref(n)),
        "select_weight_groups": lambda: L.chameleon_select_weight_groups(x, 16, bad, 1 << F.W_NF4, 1, None, x,
                                                                         x, 1 << 15, None),
        "select_pack_palette": lambda: L.chameleon_select_pack_palette(x, bad, 64, cl.PALETTE_W8,
                                                                       ctypes.byref(d), x, x, 1 << 15, x, None),
        "pack_plan": lambda: L.chameleon_pack_plan(bad, 64, x, ctypes.byref(d)),
        "pack_plan K": lambda: L.chameleon_pack_plan(16, bad, x, ctypes.byref(d)),
        "pack_plan_palette": lambda: L.chameleon_pack_plan_palette(bad, 64, cl.PALETTE_W8, ctypes.byref(d)),
        "pack_plan_grouped": lambda: L.chameleon_pack_plan_grouped(16, bad, F.W_NF4, 32, ctypes.byref(d)),
        "linear_workspace_size": lambda: L.chameleon_linear_workspace_size(bad, ctypes.byref(good), 1,
                                                                           ctypes.byref(n)),
        "linear_prepare": lambda: L.chameleon_linear_prepare(x, bad, dp, 1, x, 1 << 15, x, None),
        "linear_prepare_static": lambda: L.chameleon_linear_prepare_static(x, bad, dp, 1, ctypes.byref(p), x,
                                                                           1 << 15, x, None),
        "linear_prepare_groups": lambda: L.chameleon_linear_prepare_groups(x, bad, dp, 1, 1, x, 1 << 15, x, None),
        "linear": lambda: L.chameleon_linear(x, bad, ctypes.byref(good), x, 1, None, x, x, 1 << 15, x, None),
        "linear_gemm": lambda: L.chameleon_linear_gemm(x, bad, ctypes.byref(good), x, 1, None, x, x, 1 << 15, x,
                                                       None),
        "linear_gemm_ex": lambda: L.chameleon_linear_gemm_ex(x, bad, ctypes.byref(good), x, 1, 1, None, x,
                                                             cl.Y_F32, x, 1 << 15, x, None),
    }
    calls["act_moments_workspace_size"] = lambda: L.chameleon_act_moments_workspace_size(bad, ctypes.byref(n))
    for name, call in calls.items():
        assert call() == cl.ERR_INVALID_ARG, name


@host_buffers_only
def test_misaligned_device_pointers_are_rejected_on_the_host(cl):
    """Device pointers must be 16-byte aligned: inputs, outputs and workspaces two bytes off a
    16-byte boundary give CHAM_ERR_INVALID_ARG before any device work."""
    L = cl.lib()
    dp = ctypes.byref(cl.pack_plan(64, 64, np.zeros(64, np.uint8)))  # a 64-input layer for the prepare calls
    buf = ctypes.create_string_buffer(1 << 16)
    a = ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16
    x, m = ctypes.c_void_p(a), ctypes.c_void_p(a + 2)
    good = cl.pack_plan(64, 64, np.zeros(64, np.uint8))
    p = cl.scale_zp(F.A_E4M3, -1.0, 1.0)
    pw4 = 1 << F.W_NF4
    calls = {
        "act_moments X": lambda: L.chameleon_act_moments(m, 1024, x, x, 1 << 15, None),
        "act_quant X": lambda: L.chameleon_act_quant(m, 16, 64, 1, x, 1 << 15, x, 1 << 15, x, None),
        "act_quant qact": lambda: L.chameleon_act_quant(x, 16, 64, 1, m, 1 << 15, x, 1 << 15, x, None),
        "act_quant ws": lambda: L.chameleon_act_quant(x, 16, 64, 1, x, 1 << 15, m, 1 << 15, x, None),
        "act_quant_noalloc X": lambda: L.chameleon_act_quant_noalloc(m, 16, 64, 1, x, 1 << 15, x, None),
        "act_quant_static X": lambda: L.chameleon_act_quant_static(m, 16, 64, 1, ctypes.byref(p), x, 1 << 15, x,
                                                                   None),
        "act_quant_static qact": lambda: L.chameleon_act_quant_static(x, 16, 64, 1, ctypes.byref(p), m, 1 << 15,
                                                                      x, None),
        "act_format_sse X": lambda: L.chameleon_act_format_sse(m, 16, 64, x, x, 1 << 15, x, None),
        "act_format_sse ws": lambda: L.chameleon_act_format_sse(x, 16, 64, x, m, 1 << 15, x, None),
        "act_channel_energy X": lambda: L.chameleon_act_channel_energy(m, 16, 64, x, None),
        "select_weight_formats W": lambda: L.chameleon_select_weight_formats(m, 16, 64, cl.PALETTE_W8, x, None,
                                                                             None),
        "select_weight_groups W": lambda: L.chameleon_select_weight_groups(m, 16, 64, pw4, 1, None, x, x, 1 << 15,
                                                                           None),
        "select_weight_groups ws": lambda: L.chameleon_select_weight_groups(x, 16, 64, pw4, 1, None, x, m,
                                                                            1 << 15, None),
        "pack_weights W": lambda: L.chameleon_pack_weights(m, x, ctypes.byref(good), x, 1 << 15, x, None),
        "pack_weights blob": lambda: L.chameleon_pack_weights(x, x, ctypes.byref(good), m, 1 << 15, x, None),
        "select_pack_palette W": lambda: L.chameleon_select_pack_palette(m, 64, 64, cl.PALETTE_W8,
                                                                         ctypes.byref(good), x, x, 1 << 15, x, None),
        "select_pack_palette blob": lambda: L.chameleon_select_pack_palette(x, 64, 64, cl.PALETTE_W8,
                                                                            ctypes.byref(good), x, m, 1 << 15, x,
                                                                            None),
        "linear_prepare X": lambda: L.chameleon_linear_prepare(m, 16, dp, 1, x, 1 << 15, x, None),
        "linear_prepare ws": lambda: L.chameleon_linear_prepare(x, 16, dp, 1, m, 1 << 15, x, None),
        "linear_prepare_static X": lambda: L.chameleon_linear_prepare_static(m, 16, dp, 1, ctypes.byref(p), x,
                                                                             1 << 15, x, None),
        "linear_gemm_ex blob": lambda: L.chameleon_linear_gemm_ex(x, 16, ctypes.byref(good), m, 1, 1, None, x,
                                                                  cl.Y_F32, x, 1 << 15, x, None),
        "linear_gemm_ex Y": lambda: L.chameleon_linear_gemm_ex(x, 16, ctypes.byref(good), x, 1, 1, None, m,
                                                               cl.Y_F32, x, 1 << 15, x, None),
        "linear_gemm_ex ws": lambda: L.chameleon_linear_gemm_ex(x, 16, ctypes.byref(good), x, 1, 1, None, x,
                                                                cl.Y_F32, m, 1 << 15, x, None),
        "linear_gemm_ex bias": lambda: L.chameleon_linear_gemm_ex(x, 16, ctypes.byref(good), x, 1, 1, m, x,
                                                                  cl.Y_F32, x, 1 << 15, x, None),
        "linear_gemm_ex X (fp16 operand)": lambda: L.chameleon_linear_gemm_ex(m, 16, ctypes.byref(good), x,
                                                                              F.A_FP16, 1, None, x, cl.Y_F32, x,
                                                                              1 << 15, x, None),
    }
    for name, call in calls.items():
        assert call() == cl.ERR_INVALID_ARG, name


@host_buffers_only
def test_undersized_buffers_are_rejected_on_the_host(cl):
    """A buffer one byte smaller than its size query returned gives CHAM_ERR_WORKSPACE before any
    device work: quantized activations, workspaces, weight blobs."""
    L = cl.lib()
    dp = ctypes.byref(cl.pack_plan(64, 64, np.zeros(64, np.uint8)))  # a 64-input layer for the prepare calls
    buf = ctypes.create_string_buffer(1 << 20)
    x = ctypes.c_void_p(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 256)
    good = cl.pack_plan(64, 64, np.zeros(64, np.uint8))
    p = cl.scale_zp(F.A_E4M3, -1.0, 1.0)
    q, w = cl.act_quant_size(16, 64, F.A_E4M3)
    n = ctypes.c_size_t(0)

    def size(fn, *args):
        assert fn(*args, ctypes.byref(n)) == cl.OK
        return n.value

    sse = size(L.chameleon_act_format_sse_workspace_size, 16, 64)
    sg = size(L.chameleon_select_weight_groups_workspace_size, 16, 64, 1 << F.W_NF4, 1)
    lw = size(L.chameleon_linear_workspace_size, 16, ctypes.byref(good), F.A_E4M3)
    mw = size(L.chameleon_act_moments_workspace_size, 1024)
    e4, nf4, blob = F.A_E4M3, 1 << F.W_NF4, good.bytes
    calls = {
        "act_quant qact": lambda: L.chameleon_act_quant(x, 16, 64, e4, x, q - 1, x, w, x, None),
        "act_quant ws": lambda: L.chameleon_act_quant(x, 16, 64, e4, x, q, x, w - 1, x, None),
        "act_quant_static qact": lambda: L.chameleon_act_quant_static(x, 16, 64, e4, ctypes.byref(p), x, q - 1, x,
                                                                      None),
        "act_quant_noalloc qact": lambda: L.chameleon_act_quant_noalloc(x, 16, 64, e4, x, q - 1, x, None),
        "act_format_sse ws": lambda: L.chameleon_act_format_sse(x, 16, 64, x, x, sse - 1, x, None),
        "act_moments ws": lambda: L.chameleon_act_moments(x, 1024, x, x, mw - 1, None),
        "select_weight_groups ws": lambda: L.chameleon_select_weight_groups(x, 16, 64, nf4, 1, None, x, x, sg - 1,
                                                                            None),
        "pack_weights blob": lambda: L.chameleon_pack_weights(x, x, ctypes.byref(good), x, blob - 1, x, None),
        "select_pack_palette blob": lambda: L.chameleon_select_pack_palette(x, 64, 64, cl.PALETTE_W8,
                                                                            ctypes.byref(good), x, x, blob - 1, x,
                                                                            None),
        "linear_prepare ws": lambda: L.chameleon_linear_prepare(x, 16, dp, e4, x, lw - 1, x, None),
        "linear_prepare_static ws": lambda: L.chameleon_linear_prepare_static(x, 16, dp, e4, ctypes.byref(p), x,
                                                                              lw - 1, x, None),
        "linear_prepare_groups ws": lambda: L.chameleon_linear_prepare_groups(x, 16, dp, e4, 2, x, lw - 1, x,
                                                                              None),
        "linear_gemm ws": lambda: L.chameleon_linear_gemm(x, 16, ctypes.byref(good), x, e4, None, x, x, lw - 1, x,
                                                          None),
        "linear ws": lambda: L.chameleon_linear(x, 16, ctypes.byref(good), x, e4, None, x, x, lw - 1, x, None),
    }
    for name, call in calls.items():
        assert call() == cl.ERR_WORKSPACE, name


@host_buffers_only
def test_binding_rejects_strided_mistyped_and_host_tensors(cl):
    """The binding hands the library one dense CUDA buffer per tensor: a host tensor, a
    non-contiguous view or a tensor of the wrong element type raises in Python, before the library
    is called (element type first, then layout, then device)."""
    import torch
    X = torch.zeros(64, 32, dtype=torch.float16)
    with pytest.raises(ValueError, match="CUDA"):
        cl.act_quant(X, F.A_E4M3)                                       # a host tensor
    with pytest.raises(TypeError, match="float16"):
        cl.act_quant(X.float(), F.A_E4M3)
    with pytest.raises(TypeError, match="float16"):
        cl.select_weight_formats(torch.zeros(16, 64, dtype=torch.bfloat16), cl.PALETTE_W8)
    with pytest.raises(ValueError, match="contiguous"):
        cl._ptr(X.t())                                                  # 32 x 64 transposed view
    with pytest.raises(TypeError, match="float32"):
        cl._f32(torch.zeros(64, dtype=torch.float64), "bias")
    with pytest.raises(TypeError, match="float32"):
        cl._f32(torch.zeros(16, 64, dtype=torch.float16), "Y")
    assert cl._f32(None, "bias") is None


def test_linear_workspace_holds_the_operands_the_tiles_need(cl):
    """The workspace layout of include/chameleon.h: class-0 tiles of a 4-bit per-channel layout
    against E4M3 / E5M2 / MXFP8 activations take the 1-byte codes (M x K; MXFP8 adds its exponents
    chunk-major, ceil(K/128) x round_up(M, 4) x 4 bytes); every other tile takes the exact fp16
    operand (2 M x K); f16_only = 1 sends every tile to the fp16 path.  Differences against the
    CHAM_A_FP16 size (which holds no operand and no range partials) isolate the operand regions;
    no launch of this shape splits K (no partial sums)."""
    M, K, N = 8192, 640, 1280

    def r256(n):
        return -(-n // 256) * 256

    parts = r256(max(min(-(-(M * K // 8) // 2048), 152 * 8), 64) * 16)  # range partials, 152 SMs
    codes, fp16 = r256(M * K), r256(2 * M * K)
    e8 = r256(-(-K // 128) * -(-M // 4) * 4 * 4)
    c0 = cl.pack_plan(N, K, np.full(N, F.W_INT4_ASYM, np.uint8))
    mixed = cl.pack_plan(N, K, np.array([F.W_MXFP4, F.W_NF4] * (N // 2), np.uint8))
    w8 = cl.pack_plan(N, K, np.full(N, F.W_INT8_SYM, np.uint8))

    def extra(d, af, f16_only=0):
        d.f16_only = f16_only
        return cl.linear_workspace_size(M, d, af) - cl.linear_workspace_size(M, d, F.A_FP16)

    for af in (F.A_E4M3, F.A_E5M2):
        assert extra(c0, af) == parts + codes
        assert extra(c0, af, 1) == parts + fp16
        assert extra(mixed, af) == parts + codes + fp16
        assert extra(w8, af) == parts + fp16
    assert extra(c0, F.A_MXFP8) == parts + codes + e8
    assert extra(mixed, F.A_MXFP8) == parts + codes + e8 + fp16
    for af in (F.A_INT8_ASYM, F.A_MXINT8):
        assert extra(c0, af) == parts + fp16 and extra(mixed, af) == parts + fp16
    g = cl.pack_plan_grouped(N, K, F.W_INT4_ASYM, 64)                  # group-wise blobs: fp16 path
    assert extra(g, F.A_E4M3) == parts + fp16
    c0.f16_only = 2
    with pytest.raises(cl.ChameleonError):
        cl.linear_workspace_size(M, c0, F.A_E4M3)


def test_format_group_layout_tile_counts(cl):
    """chameleon_pack_plan_layout: layout 0 pads each MMA class to whole tiles; layout 1 pads each
    format of a class (palette order) and, with fold, the class's tail of small formats."""
    counts = {F.W_INT4_ASYM: 922, F.W_NF4: 996, F.W_E2M1: 1, F.W_MXINT4: 8, F.W_MXFP4: 2681}
    fmt = np.concatenate([np.full(n, f, np.uint8) for f, n in counts.items()])
    N, K = len(fmt), 1152
    tiles = lambda n: -(-n // 128)
    d0 = cl.pack_plan(N, K, fmt)
    assert list(d0.n_tiles) == [tiles(922 + 1 + 8 + 2681), tiles(996)] and d0.layout == 0
    d1 = cl.pack_plan(N, K, fmt, 1, 0)
    assert list(d1.n_tiles) == [tiles(922) + tiles(1) + tiles(8) + tiles(2681), tiles(996)]
    d2 = cl.pack_plan(N, K, fmt, 1, 64)
    assert list(d2.n_tiles) == [tiles(922) + tiles(2681) + tiles(1 + 8), tiles(996)]
    assert (d2.layout, d2.fold) == (1, 64) and d2.bytes > d0.bytes
    for bad in ((2, 0), (-1, 0), (1, -1)):
        with pytest.raises(cl.ChameleonError):
            cl.pack_plan(N, K, fmt, *bad)

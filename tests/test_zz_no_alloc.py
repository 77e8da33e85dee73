"""chameleon_act_quant_noalloc: the activation quantizer for callers that cannot allocate device
memory at call time (plugins of a host application or inference runtime that owns every buffer).
It must give exactly what chameleon_act_quant gives, on consecutive calls that share its static
scratch array.  Collected last on purpose (file name), and self-contained so it also passes alone
in a fresh process."""
import numpy as np
import pytest

from gpu_common import lib_module, cuda, host

pytestmark = pytest.mark.gpu


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    import torch
    cl = lib_module()
    g = np.random.default_rng(20260099)
    # the second tensor has a much smaller range: a stale partial from the first call would show
    first = (g.standard_t(3, (1024, 1280)) * 40.0).astype(np.float16)
    second = (g.standard_t(5, (333, 640)) * 0.01).astype(np.float16)
    for fmt in range(5):
        for X in (first, second):
            Xd = cuda(X)
            M, K = X.shape
            ref, st_ref = cl.act_quant(Xd, fmt)
            qb, _ = cl.act_quant_size(M, K, fmt)
            out = torch.full((qb,), 0xAB, dtype=torch.uint8, device=Xd.device)
            st = torch.zeros(1, dtype=torch.int32, device=Xd.device)
            assert cl.act_quant_noalloc(Xd, fmt, out, st) == cl.OK
            torch.cuda.synchronize()
            assert int(st.item()) == 0 and int(st_ref.item()) == 0
            c_ref, p_ref, e_ref = cl.split_qact(ref, M, K)
            c_got, p_got, e_got = cl.split_qact(out, M, K)
            np.testing.assert_array_equal(host(c_got), host(c_ref))
            assert p_got == p_ref
            if fmt >= 3:
                np.testing.assert_array_equal(host(e_got), host(e_ref))


def test_noalloc_rejects_bad_arguments():
    import torch
    cl = lib_module()
    X = torch.zeros((4, 48), dtype=torch.float16, device="cuda")
    out = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert cl.act_quant_noalloc(X, 1, out, st) == cl.ERR_INVALID_ARG        # K not a multiple of 32
    X = torch.zeros((64, 64), dtype=torch.float16, device="cuda")
    assert cl.act_quant_noalloc(X, 1, out[:16], st) == cl.ERR_WORKSPACE     # output buffer too small


def test_noalloc_reports_nonfinite_input_and_takes_exactly_sized_outputs():
    """An Inf in X reaches the caller's status word as CHAM_ERR_NONFINITE for every format, and an
    output buffer of exactly the size act_quant_size gives is accepted for shapes whose M * K is not
    a multiple of 256 (the parameter and exponent regions then start at rounded offsets)."""
    import torch
    cl = lib_module()
    g = np.random.default_rng(20260101)
    for M, K in [(3, 32), (7, 96), (333, 640)]:
        X = (g.standard_normal((M, K)) * 0.5).astype(np.float16)
        for fmt in range(5):
            qb, _ = cl.act_quant_size(M, K, fmt)
            Xd = cuda(X)
            out = torch.empty((qb,), dtype=torch.uint8, device=Xd.device)
            st = torch.zeros(1, dtype=torch.int32, device=Xd.device)
            assert cl.act_quant_noalloc(Xd, fmt, out, st) == cl.OK
            ref, st_ref = cl.act_quant(Xd, fmt)
            torch.cuda.synchronize()
            assert int(st.item()) == 0 and int(st_ref.item()) == 0
            np.testing.assert_array_equal(host(cl.split_qact(out, M, K)[0]), host(cl.split_qact(ref, M, K)[0]))
            bad = X.copy()
            bad[M // 2, K - 1] = np.float16(np.inf)
            st.zero_()
            assert cl.act_quant_noalloc(cuda(bad), fmt, out, st) == cl.OK
            torch.cuda.synchronize()
            assert int(st.item()) == cl.ERR_NONFINITE, (M, K, fmt)

"""Failure detection without a GPU fault: a GEMM whose producer withholds one K-chunk (a barrier
that nothing completes) must end on its own with CHAM_ERR_TIMEOUT in the device status word, and
the context must stay usable (the next call is correct)."""
import time

import numpy as np
import pytest

from oracle import formats as F
from oracle import gemm as G
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host, assert_within_bound

pytestmark = pytest.mark.gpu


def test_withheld_chunk_times_out_and_context_survives():
    import torch
    cl = lib_module()
    X, W, bias = WL.single_layer(M=256, K=640, N=256)
    fmt = np.full(W.shape[0], F.W_INT8_SYM, np.uint8)
    d = cl.pack_plan(W.shape[0], W.shape[1], fmt)
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    Xd, bd = cuda(X), cuda(bias)
    cl.debug_stall_next_gemm(1)   # CTA 0 owns at least two K-chunks, with or without split-K
    t0 = time.time()
    Y, st2 = cl.linear(Xd, d, blob, F.A_E4M3, bias=bd)
    torch.cuda.synchronize()
    assert int(st2.item()) == cl.ERR_TIMEOUT
    assert time.time() - t0 < 30.0
    Y, st3 = cl.linear(Xd, d, blob, F.A_E4M3, bias=bd)  # one-shot hook: this call is normal
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st3.item()) == 0
    Y_ref, bound, _, _ = G.linear_reference(X, F.A_E4M3, W, fmt, bias)
    assert_within_bound(host(Y), Y_ref, bound, "after a timed-out call")

"""Pins of the oracle's fp64 linear reference: special operands with known exact products and a
triple-loop re-computation on tiny sizes."""
import numpy as np

from oracle import formats as F
from oracle import gemm as G

RNG = np.random.default_rng(20260020)


def test_identity_weights_give_dequantized_activations():
    """W = I in a format whose DQ(I) is exactly I (MXINT8: block max 1 -> X = 0, code 64;
    NF4: s = 1, level 15 = 1; MXFP4: X = -2, code 4.0): Y = DQ(A) exactly."""
    K = 64
    X = (RNG.standard_t(3, (8, K)) * 0.5).astype(np.float16)
    Wt = np.eye(K, dtype=np.float16)
    for wf in (F.W_MXINT8, F.W_NF4, F.W_MXFP4, F.W_MXINT4):
        for af in F.ACT_FORMATS:
            y, bound, a, w = G.linear_reference(X, af, Wt, np.full(K, wf, np.uint8))
            np.testing.assert_array_equal(w, np.eye(K))
            np.testing.assert_array_equal(y, a)


def test_one_hot_rows_select_weight_columns():
    K, N = 64, 48
    X = np.zeros((K, K), np.float16)
    X[np.arange(K), np.arange(K)] = 1.0                      # MXINT8: DQ(one-hot) = one-hot
    W = RNG.normal(0, 0.02, (N, K)).astype(np.float16)
    wf = RNG.choice([F.W_INT4_SYM, F.W_NF4, F.W_E2M1, F.W_MXFP4], N).astype(np.uint8)
    bias = RNG.normal(0, 0.02, N)
    y, _, a, w = G.linear_reference(X, F.A_MXINT8, W, wf, bias)
    np.testing.assert_array_equal(a, np.eye(K))
    np.testing.assert_array_equal(y, w.T + bias[None, :])


def test_against_triple_loop():
    M, K, N = 5, 64, 7
    X = (RNG.standard_t(3, (M, K)) * 0.5).astype(np.float16)
    W = RNG.normal(0, 0.02, (N, K)).astype(np.float16)
    wf = RNG.choice(range(3), N).astype(np.uint8)
    bias = RNG.normal(0, 0.02, N)
    for af in F.ACT_FORMATS:
        y, bound, a, w = G.linear_reference(X, af, W, wf, bias)
        for m in range(M):
            for n in range(N):
                acc = 0.0
                acc_abs = 0.0
                for k in range(K):
                    acc += a[m, k] * w[n, k]
                    acc_abs += abs(a[m, k] * w[n, k])
                assert abs(y[m, n] - (acc + bias[n])) <= 1e-12
                assert abs(bound[m, n] - 2.0 ** -10 * acc_abs) <= 1e-15


def test_fp16_passthrough_for_weight_only_fork():
    X = RNG.normal(0, 1, (4, 64)).astype(np.float16)
    W = RNG.normal(0, 0.02, (6, 64)).astype(np.float16)
    y, _, a, _ = G.linear_reference(X, F.A_FP16, W, np.full(6, F.W_NF4, np.uint8))
    np.testing.assert_array_equal(a, X.astype(np.float64))

"""Helpers shared by the GPU parity tests: build/load the library, move arrays, compare."""
import numpy as np
import pytest


def lib_module():
    """The binding with the library built for this machine; fails (never falls back) without one."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2609_33496_gb300 import build
    build.build()
    import paper_2609_33496_gb300 as P
    P.chameleon.lib()
    return P.chameleon


def cuda(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.detach().cpu().numpy()


def assert_within_bound(Y, Y_ref, bound, what=""):
    err = np.abs(Y.astype(np.float64) - Y_ref)
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError("%s: %d / %d outside 2^-10 sum|a w| (first at %s: got %r ref %r bound %r)"
                             % (what, int(bad.sum()), bad.size, tuple(i), float(Y[tuple(i)]),
                                float(Y_ref[tuple(i)]), float(bound[tuple(i)])))

"""GPU calibration power sums (Alg. 1 accumulator) and kurtosis against the oracle."""
import numpy as np
import pytest

from oracle import schedule as S
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def test_moments_and_kurtosis(cl):
    import torch
    out = None
    xs = [WL.sdxl_layer_activation(0, b, rows=512) for b in (0, 5, 9)]
    for X in xs:
        out = cl.act_moments(cuda(X), out)
    torch.cuda.synchronize()
    got = host(out)
    ref = S.power_sums(np.concatenate([x.astype(np.float64).ravel() for x in xs]))
    assert got[0] == ref["n"]
    for i, k in enumerate(("s1", "s2", "s3", "s4")):
        assert got[1 + i] == pytest.approx(ref[k], rel=1e-10, abs=1e-6)
    assert got[5] == ref["lo"] and got[6] == ref["hi"]
    assert cl.kurtosis(got[:5]) == pytest.approx(S.kurtosis_from_sums(*[ref[k] for k in ("n", "s1", "s2", "s3", "s4")]),
                                                 rel=1e-9)

"""Failure detection on the GPU without a GPU fault: a wait that is never
satisfied (an mbarrier nothing arrives at, a group barrier one CTA never
reaches) must give up after its limit of about a second, report
SLS_ERR_TIMEOUT through the status word, and leave the context usable."""
import time

import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import feature_tolerance, to_torch_x

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


@pytest.mark.parametrize("which", [0, 1])
def test_stuck_wait_ends_with_timeout_status(sls, which):
    t0 = time.time()
    st = sls.selftest_wait_limit(which)
    elapsed = time.time() - t0
    assert st == 5, st                      # SLS_ERR_TIMEOUT
    assert elapsed < 30.0, elapsed          # about one second of clock cycles
    # the context still works: a small feature map against the oracle
    w = WL.scaled(WL.WORKLOADS["tiny"], N=200, D=256)
    p, prm = WL.make_prompt(w), WL.params_for(w)
    phi = sls.feature_map(to_torch_x(p.X, w.dtype), to_torch_x(prm.W, w.dtype),
                          torch.from_numpy(prm.b).cuda())
    got = phi.cpu().numpy().astype(np.float64)
    want = O.rff_features(p.x_f64(), prm.w_f64(), prm.b)
    assert np.all(np.abs(got - want) <= feature_tolerance(p.x_f64(), prm.w_f64(),
                                                          prm.b.astype(np.float64)))

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


def test_lanczos_giveup_leaves_empty_result_and_usable_context(sls):
    """The persistent Lanczos kernel's own give-up path: one CTA reports a
    failed wait at its first group barrier (as a wait that ran out would), so
    the group is released, the copy warps stop after their bounded wait, the
    status reads SLS_ERR_TIMEOUT, r_eff stays -1 and the later kernels treat
    the problem as empty (theta and U zero) instead of reading stale values.
    The same problem then runs normally and matches the oracle."""
    g = np.random.default_rng(5)
    N, D, r = 3000, 512, 24
    X = g.standard_normal((N, 24)) / np.sqrt(24)
    W = g.standard_normal((D, 24)) * 24 ** -0.25
    b = g.random(D) * 2 * np.pi
    phi32 = O.rff_features(X, W, b).astype(np.float32)
    q1 = g.standard_normal(N)
    Phi, Q1 = torch.from_numpy(phi32).cuda(), torch.from_numpy(q1).cuda()
    t0 = time.time()
    status, theta, U, r_eff = sls.selftest_lanczos_giveup(Phi, Q1, r)
    torch.cuda.synchronize()
    assert time.time() - t0 < 30.0
    assert status == 5, status
    assert int(r_eff.item()) == -1
    assert float(theta.abs().max().item()) == 0.0
    assert float(U.abs().max().item()) == 0.0
    # the context still works, and a normal call gives the oracle's result
    th, U2, k, _, _ = sls.lanczos_topr(Phi, Q1, r)
    a, be, Q, ko = O.lanczos(phi32.astype(np.float64), q1, r)
    th_o, _, U_o = O.ritz_pairs(a, be, Q)
    assert int(k.item()) == ko
    t = th.cpu().numpy()[:ko]
    assert np.all(np.abs(t - th_o) <= 1e-4 * np.abs(th_o) + 1e-12 * abs(th_o[0]))

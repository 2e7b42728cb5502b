"""Parity of the batched Lanczos launch -- the plan sls_compress uses for the
windows of its adaptive and local backends -- against the oracle, window by
window (Algorithm 2 per window, Sec. 3.5-3.6).

In that plan the persistent kernel's CTAs form groups, each group runs one
window at a time on a strip of rows per CTA, and a group takes the next
window as soon as it finishes one.  The windows here have the adaptive
workload's shape (2048-token windows of prompts of 16384 tokens, d = 4096
bf16, D = 1024, r = 32; the last window of each prompt is ragged), enough of
them that some groups run two windows back to back, each window compared
with oracle.lanczos and oracle.ritz_pairs on the same float32 feature rows
and start vector.  A second case has many small windows with one CTA each."""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import max_subspace_angle, to_torch_x

pytestmark = pytest.mark.gpu

RITZ_RTOL = 1e-4
ANGLE_TOL = 1e-3
ZERO_FLOOR = 1e-12


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


def _check_window(theta, U, k_gpu, phi64, q1, r):
    a, be, Q, k = O.lanczos(phi64, q1, r)
    th_o, _, U_o = O.ritz_pairs(a, be, Q)
    assert k_gpu == k
    th = theta[:k]
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + ZERO_FLOOR * abs(th_o[0])), \
        float(np.max(err / np.abs(th_o)))
    ang = max_subspace_angle(U[:, :k], U_o)
    assert ang <= ANGLE_TOL, ang
    return ang


def test_lanczos_batched_adaptive_window_shape(sls):
    w = WL.WORKLOADS["adaptive"]
    prompts = list(range(0, 64, 7))        # 10 prompts, duplication 0 .. 0.6
    B, N, d, D, r, win = len(prompts), w.N, w.d, w.D, w.r, w.window
    Nc = N - w.preserve_last
    Xs = [WL.make_prompt(w, index=i, dup_frac=WL.adaptive_dup_frac(i, w.batch)).X
          for i in prompts]
    X = to_torch_x(np.stack(Xs), "bf16")
    prm = WL.params_for(w)
    W = to_torch_x(prm.W, "bf16")
    b = torch.from_numpy(prm.b).cuda()
    # the feature map launch sls_compress makes (one launch over the batch)
    phi = sls.feature_map_batched(X, W, b, Nc)
    row0, n, q1off = [], [], []
    for k in range(B):
        for s in range(0, Nc, win):
            row0.append(k * Nc + s)
            n.append(min(win, Nc - s))
            q1off.append(k * N + s)
    assert len(n) == 8 * B and n[7] == Nc - 7 * win   # 7 full windows + 1 ragged
    q1 = prm.q1[:B * N]
    theta, U, r_eff, _, _ = sls.lanczos_topr_batched(phi, torch.from_numpy(q1).cuda(), r,
                                                     row0, n, q1off)
    torch.cuda.synchronize()
    theta, U, r_eff = theta.cpu().numpy(), U.cpu().numpy(), r_eff.cpu().numpy()
    phi_h = phi.cpu().numpy()
    worst = 0.0
    for p, (r0, nn, qo) in enumerate(zip(row0, n, q1off)):
        ang = _check_window(theta[p], U[r0:r0 + nn], int(r_eff[p]),
                            phi_h[r0:r0 + nn].astype(np.float64), q1[qo:qo + nn], r)
        worst = max(worst, ang)
    print(f"batched adaptive-shape Lanczos: {len(n)} windows, max subspace angle {worst:.2e}")


def test_lanczos_batched_many_small_windows(sls):
    """More windows than CTA groups (one CTA per window): groups run several
    windows back to back; ragged window lengths."""
    g = np.random.default_rng(11)
    D, r, nprob = 256, 16, 200
    n = g.integers(200, 301, size=nprob)
    row0 = np.concatenate([[0], np.cumsum(n)[:-1]])
    rows = int(n.sum())
    X = g.standard_normal((rows, 16)) / 4.0
    Wm = g.standard_normal((D, 16)) * 16 ** -0.25
    bb = g.random(D) * 2 * np.pi
    phi32 = O.rff_features(X, Wm, bb).astype(np.float32)
    q1 = g.standard_normal(rows)
    theta, U, r_eff, _, _ = sls.lanczos_topr_batched(torch.from_numpy(phi32).cuda(),
                                                     torch.from_numpy(q1).cuda(), r,
                                                     row0, n)
    torch.cuda.synchronize()
    theta, U, r_eff = theta.cpu().numpy(), U.cpu().numpy(), r_eff.cpu().numpy()
    for p in range(nprob):
        r0, nn = int(row0[p]), int(n[p])
        _check_window(theta[p], U[r0:r0 + nn], int(r_eff[p]),
                      phi32[r0:r0 + nn].astype(np.float64), q1[r0:r0 + nn], r)

"""The feature matrix stored in bfloat16 (opt-in half-size Phi): the feature
map's bf16 output against the oracle's features, and Lanczos on bf16 rows
against the oracle's Lanczos on the same rounded values, at the float32
path's bars (Ritz values 1e-4 relative, subspace angle 1e-3 rad); the
whole pass with bf16 storage by its invariants and the oracle's macro
embeddings of the GPU's own groups."""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import feature_tolerance, max_subspace_angle, oracle_phi32, to_torch_x

pytestmark = pytest.mark.gpu

RITZ_RTOL = 1e-4
ANGLE_TOL = 1e-3
ZERO_FLOOR = 1e-12
EMB_TOL = 1e-4


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


def _inputs(name, N, D, d=None):
    w = WL.scaled(WL.WORKLOADS[name], N=N, D=D, d=d or WL.WORKLOADS[name].d)
    return w, WL.make_prompt(w), WL.params_for(w)


def _bf16_tensor(x64):
    """float64 values already on the bf16 grid -> a CUDA bfloat16 tensor."""
    bits = WL.f32_to_bf16_bits(np.asarray(x64, dtype=np.float32))
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()


def _widen(t):
    return t.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("name,N,D", [("tiny", 500, 256), ("mistral7b", 700, 1024),
                                      ("mistral7b", 333, 2048)])
def test_feature_map_bf16_output(sls, name, N, D):
    """Each stored feature is the bf16 rounding of a value within the float32
    path's bound of the oracle's float64 feature."""
    w, p, prm = _inputs(name, N, D)
    X64, W64, b = p.x_f64(), prm.w_f64(), prm.b
    phi = sls.feature_map(to_torch_x(p.X, w.dtype), to_torch_x(prm.W, w.dtype),
                          torch.from_numpy(b).cuda(), phi_dtype=torch.bfloat16)
    assert phi.dtype == torch.bfloat16 and tuple(phi.shape) == (N, D)
    got = _widen(phi)
    want = O.rff_features(X64, W64, b)
    tol = feature_tolerance(X64, W64, b.astype(np.float64))
    half_ulp = 2.0 ** -8 * np.maximum(np.abs(got), np.abs(want))
    assert np.all(np.abs(got - want) <= tol + half_ulp)
    # got is on the bf16 grid, and it is the rounding of the oracle's value
    # except where the float32 evaluation straddles a rounding boundary
    assert np.array_equal(O.bf16_round(got), got)
    assert np.mean(got == O.bf16_round(want)) > 0.99


def _lanczos_bf16_case(sls, phib64, q1, r):
    theta, U, r_eff, alpha, beta = sls.lanczos_topr(_bf16_tensor(phib64),
                                                    torch.from_numpy(q1).cuda(), r)
    torch.cuda.synchronize()
    a, b_, Q, k = O.lanczos(phib64, q1, r)
    th_o, S_o, U_o = O.ritz_pairs(a, b_, Q)
    assert int(r_eff.item()) == k
    th = theta.cpu().numpy()[:k]
    floor = ZERO_FLOOR * abs(th_o[0])
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + floor), float(np.max(err / np.abs(th_o)))
    assert max_subspace_angle(U.cpu().numpy()[:, :k], U_o) <= ANGLE_TOL
    return th, th_o


@pytest.mark.parametrize("name,N,D,r", [("tiny", 500, 256, 16),      # narrow D: row phases
                                        ("mistral7b", 8180, 1024, 32),
                                        ("mistral7b", 3001, 2048, 64),  # two groups per thread
                                        ("tiny", 16, 256, 8),        # window kernel
                                        ("tiny", 29, 64, 8)])
def test_lanczos_bf16_phi_matches_oracle(sls, name, N, D, r):
    w, p, prm = _inputs(name, N, D)
    phib = O.bf16_round(oracle_phi32(p.x_f64(), prm.w_f64(), prm.b).astype(np.float64))
    th, th_o = _lanczos_bf16_case(sls, phib, prm.q1[:N], r)
    # the tolerance class of bf16 storage: the leading Ritz value within the
    # Weyl bound (2u + u^2) |Phi|^2 of the float32 operator's (u = 2^-8)
    phi = oracle_phi32(p.x_f64(), prm.w_f64(), prm.b).astype(np.float64)
    a, b_, Q, k = O.lanczos(phi, prm.q1[:N], r)
    th32 = O.ritz_pairs(a, b_, Q)[0]
    u = 2.0 ** -8
    assert abs(th[0] - th32[0]) <= (2 * u + u * u) * np.linalg.norm(phi, 2) ** 2


def test_lanczos_bf16_rejects_unaligned_width(sls):
    phib = O.bf16_round(np.random.default_rng(0).standard_normal((40, 12)) * 0.1)
    with pytest.raises(sls.SLSError):
        sls.lanczos_topr(_bf16_tensor(phib), torch.ones(40, dtype=torch.float64).cuda(), 4)


def _check_groups(X64, Xt, pos, t2m, M, pl):
    N = X64.shape[0]
    t2m = t2m.astype(np.int64)
    assert t2m.min() == 0 and t2m.max() == M - 1
    assert np.all(np.bincount(t2m, minlength=M) >= 1)
    for i in range(pl):
        assert t2m[N - pl + i] == M - pl + i and pos[M - pl + i] == N - pl + i
    groups = [np.nonzero(t2m == m)[0] for m in range(M)]
    assert np.max(np.abs(Xt - O.aggregate_groups(X64, groups, True))) <= EMB_TOL
    assert np.array_equal(pos, [O.group_position(g, O.POS_MAX) for g in groups])
    assert np.all(np.diff(pos) > 0)


@pytest.mark.parametrize("backend", ["global", "local", "adaptive"])
def test_compress_bf16_phi(sls, backend):
    w, p, prm = _inputs("mistral7b", 1500, 256, d=128)
    kw = dict(rho=8.0, D=256, r=16, bits=10, preserve_last=12, phi_dtype=sls.SLS_BF16)
    if backend == "local":
        kw.update(backend=sls.BACKEND_LOCAL, window=16, bits=0)
    elif backend == "adaptive":
        kw.update(backend=sls.BACKEND_ADAPTIVE, window=256, bits=0, rho=16.0)
    cfg = sls.Config.make(**kw)
    Xt, pos, t2m, r_eff, route = sls.compress(
        to_torch_x(p.X, w.dtype), cfg, to_torch_x(prm.W, w.dtype),
        torch.from_numpy(prm.b).cuda(), torch.from_numpy(prm.R).cuda(),
        torch.from_numpy(prm.q1).cuda())
    torch.cuda.synchronize()
    M = sls.output_count(cfg, w.N)
    _check_groups(p.x_f64(), Xt.cpu().numpy(), pos.cpu().numpy(), t2m.cpu().numpy(), M, 12)
    if backend == "global":
        assert int(r_eff[0].item()) == 16


def test_compress_bf16_phi_rejects_normalize(sls):
    cfg = sls.Config.make(rho=4.0, D=256, r=8, normalize=1, phi_dtype=sls.SLS_BF16)
    X = torch.zeros((100, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sls.SLSError):
        sls.compress(X, cfg, torch.zeros((256, 64), dtype=torch.bfloat16, device="cuda"),
                     torch.zeros(256, device="cuda"), torch.zeros((8, 8), device="cuda"),
                     torch.ones(100, dtype=torch.float64, device="cuda"))

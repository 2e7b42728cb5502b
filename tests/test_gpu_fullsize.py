"""Parity at the benchmarked sizes: the Qwen2.5-7B-shaped prompt (N = 32768,
d = 3584 bf16, D = 2048, r = 64, b = 16, rho = 16) and the Qwen2.5-14B-shaped
prompt (N = 131072, d = 5120), in the launch configuration bench.py times.

At the 7B shape the oracle runs every stage at full size, each stage fed the
same inputs as the GPU: Ritz values and subspace of the Lanczos run on the
GPU's own float32 Phi, SimHash codes bit-exact on the oracle's U, groups,
positions and macro embeddings of the aggregation on the oracle's codes.  The
whole compression pass (and the 14B shape) is checked by sampled outputs
the oracle computes one by one and by invariants that hold at any size."""
import math

import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import feature_tolerance, max_subspace_angle, to_torch_x

pytestmark = pytest.mark.gpu

RITZ_RTOL = 1e-4
ANGLE_TOL = 1e-3
EMB_TOL = 1e-4
ZERO_FLOOR = 1e-12


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


def _inputs(name):
    w = WL.WORKLOADS[name]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    return {"w": w, "p": p, "prm": prm, "Nc": w.N - w.preserve_last,
            "X": to_torch_x(p.X, "bf16"), "W": to_torch_x(prm.W, "bf16"),
            "b": torch.from_numpy(prm.b).cuda(), "R": torch.from_numpy(prm.R).cuda(),
            "q1": torch.from_numpy(prm.q1).cuda()}


def _rows64(p, rows):
    return WL.bf16_bits_to_f32(p.X[rows]).astype(np.float64)


@pytest.fixture(scope="module")
def q7(sls):
    return _inputs("qwen7b")


@pytest.fixture(scope="module")
def q7_oracle(sls, q7):
    """The GPU feature matrix of the compressible rows and the oracle's
    Lanczos run, Ritz pairs, codes and groups on it."""
    w, prm, Nc = q7["w"], q7["prm"], q7["Nc"]
    phi = sls.feature_map(q7["X"][:Nc], q7["W"], q7["b"])
    phi64 = phi.cpu().numpy().astype(np.float64)
    a, be, Q, k = O.lanczos(phi64, prm.q1[:Nc], w.r)
    th, S, U = O.ritz_pairs(a, be, Q)
    U32 = U.astype(np.float32)
    codes = O.simhash(U32, prm.R[:w.bits, :k])
    return {"phi": phi, "theta": th, "U": U, "U32": U32, "r_eff": k, "codes": codes}


def _check_compress(sls, X64_rows, p, Xt, pos, t2m, M, N, pl, rng, nsample=256):
    """Invariants of one compressed prompt, and sampled macro embeddings and
    positions recomputed by the oracle from the GPU's own groups."""
    t2m = t2m.astype(np.int64)
    assert t2m.min() == 0 and t2m.max() == M - 1
    counts = np.bincount(t2m, minlength=M)
    assert np.all(counts >= 1)
    for i in range(pl):
        assert t2m[N - pl + i] == M - pl + i and pos[M - pl + i] == N - pl + i
    assert np.all(np.diff(pos) > 0)  # max positions: causal order, no ties
    order = np.argsort(t2m, kind="stable")
    starts = np.concatenate([[0], np.cumsum(counts)])
    for m in rng.choice(M, size=min(nsample, M), replace=False):
        mem = order[starts[m]:starts[m + 1]]
        assert pos[m] == mem.max()
        want = O.aggregate_groups(X64_rows(mem), [np.arange(len(mem))], True)[0]
        assert np.max(np.abs(Xt[m] - want)) <= EMB_TOL


def test_qwen7b_features_sampled_rows(sls, q7, q7_oracle):
    rng = np.random.default_rng(70)
    rows = np.sort(rng.choice(q7["Nc"], size=256, replace=False))
    X64 = _rows64(q7["p"], rows)
    W64, b = q7["prm"].w_f64(), q7["prm"].b
    got = q7_oracle["phi"][torch.from_numpy(rows).cuda()].cpu().numpy().astype(np.float64)
    want = O.rff_features(X64, W64, b)
    tol = feature_tolerance(X64, W64, b.astype(np.float64))
    assert np.all(np.abs(got - want) <= tol), float(np.max(np.abs(got - want) / tol))


def test_qwen7b_lanczos_full_size(sls, q7, q7_oracle):
    w, Nc = q7["w"], q7["Nc"]
    theta, U, r_eff, alpha, beta = sls.lanczos_topr(q7_oracle["phi"], q7["q1"][:Nc], w.r)
    torch.cuda.synchronize()
    k = q7_oracle["r_eff"]
    assert int(r_eff.item()) == k == w.r
    th_o = q7_oracle["theta"]
    th = theta.cpu().numpy()[:k]
    floor = ZERO_FLOOR * abs(th_o[0])
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + floor), float(np.max(err / np.abs(th_o)))
    assert max_subspace_angle(U.cpu().numpy()[:, :k], q7_oracle["U"]) <= ANGLE_TOL


def test_qwen7b_lanczos_bf16_phi_full_size(sls, q7):
    """bf16 storage of Phi at the qwen7b shape: the GPU's bf16 features (the
    feature map's bf16 epilogue) run through the bf16 Lanczos kernel, against
    the oracle's Lanczos on the same stored values."""
    w, Nc = q7["w"], q7["Nc"]
    phib = sls.feature_map(q7["X"][:Nc], q7["W"], q7["b"], phi_dtype=torch.bfloat16)
    theta, U, r_eff, _, _ = sls.lanczos_topr(phib, q7["q1"][:Nc], w.r)
    torch.cuda.synchronize()
    a, be, Q, k = O.lanczos(phib.float().cpu().numpy().astype(np.float64),
                            q7["prm"].q1[:Nc], w.r)
    th_o, S, U_o = O.ritz_pairs(a, be, Q)
    assert int(r_eff.item()) == k
    th = theta.cpu().numpy()[:k]
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + ZERO_FLOOR * abs(th_o[0]))
    assert max_subspace_angle(U.cpu().numpy()[:, :k], U_o) <= ANGLE_TOL


def test_qwen7b_simhash_full_size_bit_exact(sls, q7, q7_oracle):
    w = q7["w"]
    got = sls.simhash(torch.from_numpy(q7_oracle["U32"]).cuda(), q7["R"], w.bits)
    assert np.array_equal(got.cpu().numpy().view(np.uint32), q7_oracle["codes"])


def test_qwen7b_aggregate_full_size_bit_exact(sls, q7, q7_oracle):
    w, Nc, p = q7["w"], q7["Nc"], q7["p"]
    codes = q7_oracle["codes"]
    M = O.target_count(Nc, w.rho)
    Xt, pos, t2m = sls.aggregate(q7["X"][:Nc], torch.from_numpy(codes.view(np.int32)).cuda(), M)
    clusters = O.bucket(codes)
    groups = O.adjust_groups(clusters, M)
    order = O.order_groups(groups, O.POS_MAX)
    t2m_o = np.empty(Nc, dtype=np.int64)
    for k, i in enumerate(order):
        t2m_o[groups[i]] = k
    pos_o = np.array([O.group_position(groups[i], O.POS_MAX) for i in order])
    assert np.array_equal(t2m.cpu().numpy(), t2m_o)
    assert np.array_equal(pos.cpu().numpy(), pos_o)
    Xt = Xt.cpu().numpy()
    rng = np.random.default_rng(71)
    for m in rng.choice(M, size=256, replace=False):
        mem = groups[order[m]]
        want = O.aggregate_groups(_rows64(p, mem), [np.arange(len(mem))], True)[0]
        assert np.max(np.abs(Xt[m] - want)) <= EMB_TOL


def _compress_case(sls, name, nsample):
    d = _inputs(name)
    w, p = d["w"], d["p"]
    cfg = sls.Config.make(backend=sls.BACKEND_GLOBAL, rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                          preserve_last=w.preserve_last)
    M = sls.output_count(cfg, w.N)
    assert M == O.target_count(d["Nc"], w.rho) + w.preserve_last
    Xt, pos, t2m, r_eff, route = sls.compress(d["X"].view(1, w.N, w.d), cfg, d["W"], d["b"],
                                              d["R"], d["q1"])
    torch.cuda.synchronize()
    assert int(r_eff[0].item()) == w.r
    rng = np.random.default_rng(72)
    _check_compress(sls, lambda rows: _rows64(p, rows), p, Xt[0].cpu().numpy(),
                    pos[0].cpu().numpy(), t2m[0].cpu().numpy(), M, w.N, w.preserve_last, rng,
                    nsample)
    return d


def test_qwen7b_compress_full_size(sls):
    _compress_case(sls, "qwen7b", 256)


def test_qwen14b_compress_full_size(sls):
    _compress_case(sls, "qwen14b", 128)


@pytest.fixture(scope="module")
def q14(sls):
    """The qwen14b-shaped prompt and the GPU feature matrix of its 131060
    compressible rows from the launch sls_compress makes (one batched
    tensor-core launch over all row tiles)."""
    d = _inputs("qwen14b")
    w, Nc = d["w"], d["Nc"]
    d["phi"] = sls.feature_map_batched(d["X"].view(1, w.N, w.d), d["W"], d["b"], Nc)
    return d


def test_qwen14b_features_full_launch_sampled_rows(sls, q14):
    rng = np.random.default_rng(74)
    rows = np.sort(rng.choice(q14["Nc"], size=256, replace=False))
    got = q14["phi"][torch.from_numpy(rows).cuda()].cpu().numpy().astype(np.float64)
    X64 = _rows64(q14["p"], rows)
    W64, b = q14["prm"].w_f64(), q14["prm"].b
    want = O.rff_features(X64, W64, b)
    tol = feature_tolerance(X64, W64, b.astype(np.float64))
    assert np.all(np.abs(got - want) <= tol), float(np.max(np.abs(got - want) / tol))


def test_qwen14b_lanczos_full_size(sls, q14):
    """Algorithm 2 at the qwen14b shape (N = 131060, D = 2048, r = 64) on the
    GPU's own feature matrix against the oracle: Ritz values, the Ritz
    subspace, orthonormality of the GPU's Ritz vectors and their residuals
    |A u - theta u| against the oracle's (the persistent kernel applies one
    classical Gram-Schmidt pass per step, the oracle two)."""
    w, Nc = q14["w"], q14["Nc"]
    theta, U, r_eff, _, _ = sls.lanczos_topr(q14["phi"], q14["q1"][:Nc], w.r)
    torch.cuda.synchronize()
    phi64 = q14["phi"].cpu().numpy().astype(np.float64)
    q1 = q14["prm"].q1[:Nc]
    a, be, Q, k = O.lanczos(phi64, q1, w.r)
    th_o, _, U_o = O.ritz_pairs(a, be, Q)
    assert int(r_eff.item()) == k == w.r
    th = theta.cpu().numpy()[:k]
    floor = ZERO_FLOOR * abs(th_o[0])
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + floor), float(np.max(err / np.abs(th_o)))
    Ug = U.cpu().numpy()[:, :k].astype(np.float64)
    ang = max_subspace_angle(Ug, U_o)
    assert ang <= ANGLE_TOL, ang
    orth = float(np.max(np.abs(Ug.T @ Ug - np.eye(k))))
    assert orth <= 1e-5, orth
    # residuals of the Ritz pairs, A = Phi Phi^T applied in float64
    def resid(Um, t):
        AU = phi64 @ (phi64.T @ Um)
        return np.linalg.norm(AU - Um * t[None, :], axis=0)
    rg, ro = resid(Ug, th), resid(U_o, th_o)
    assert np.all(rg <= ro + 1e-6 * abs(th_o[0])), float(np.max(rg - ro))
    print(f"qwen14b Lanczos: max rel Ritz err {float(np.max(err / np.abs(th_o))):.2e}, "
          f"angle {ang:.2e}, |U^T U - I| {orth:.2e}, max residual gpu {rg.max():.3e} "
          f"oracle {ro.max():.3e}")

"""Parity of the CUDA path (through the C ABI) with the CPU oracle on seeded
synthetic inputs.  Bars: codes, cluster and token maps bit-exact; Ritz values
relative error <= 1e-4 with the largest principal angle between the Ritz
subspaces <= 1e-3 rad (both sides fed the same float32 Phi and q1); macro
embeddings max-abs <= 1e-4; feature map within the float32 bound of
gpu_util.feature_tolerance."""
import math

import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import feature_tolerance, max_subspace_angle, oracle_phi32, to_torch_x, widen

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


def _workload_inputs(name, N=None, d=None, D=None):
    w = WL.WORKLOADS[name]
    if N is not None or d is not None or D is not None:
        w = WL.scaled(w, N=N or w.N, d=d or w.d, D=D or w.D)
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    return w, p, prm


# ---------------------------------------------------------------------------
# feature map (Sec. 3.2)
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("name,N,D", [("tiny", 512, 256), ("mistral7b", 1000, 1024),
                                      ("qwen7b", 777, 2048)])
def test_feature_map_matches_oracle(sls, name, N, D):
    w, p, prm = _workload_inputs(name, N=N, D=D)
    X64 = p.x_f64()
    W64 = prm.w_f64()
    phi = sls.feature_map(to_torch_x(p.X, w.dtype), to_torch_x(prm.W, w.dtype),
                          torch.from_numpy(prm.b).cuda())
    got = phi.cpu().numpy().astype(np.float64)
    want = O.rff_features(X64, W64, prm.b)
    tol = feature_tolerance(X64, W64, prm.b.astype(np.float64))
    err = np.abs(got - want)
    assert np.all(err <= tol), float(np.max(err / tol))


def test_feature_map_ragged_and_empty(sls):
    g = np.random.default_rng(0)
    for N, d, D in [(1, 8, 4), (129, 40, 68), (300, 8, 260)]:
        X = g.standard_normal((N, d)).astype(np.float32) / math.sqrt(d)
        W = (g.standard_normal((D, d)) * d ** -0.25).astype(np.float32)
        b = (g.random(D) * 2 * math.pi).astype(np.float32)
        phi = sls.feature_map(torch.from_numpy(X).cuda(), torch.from_numpy(W).cuda(),
                              torch.from_numpy(b).cuda()).cpu().numpy()
        want = O.rff_features(X, W, b)
        tol = feature_tolerance(X.astype(np.float64), W.astype(np.float64), b.astype(np.float64))
        assert np.all(np.abs(phi - want) <= tol)
    out = sls.feature_map(torch.zeros((0, 8), device="cuda"), torch.zeros((4, 8), device="cuda"),
                          torch.zeros(4, device="cuda"))
    assert out.shape == (0, 4)


@pytest.mark.parametrize("N,d,D", [(300, 200, 512), (129, 8, 256), (1, 72, 256)])
def test_feature_map_tc_partial_k_tile(sls, N, d, D):
    """bf16 shapes on the tensor-core path whose d is not a multiple of the K
    tile (the last K block is zero-filled by the copy engine) and whose row
    count leaves a partial row tile."""
    g = np.random.default_rng(N + d)
    Xb = WL.f32_to_bf16_bits((g.standard_normal((N, d)) / math.sqrt(d)).astype(np.float32))
    Wb = WL.f32_to_bf16_bits((g.standard_normal((D, d)) * d ** -0.25).astype(np.float32))
    b = (g.random(D) * 2 * math.pi).astype(np.float32)
    X64, W64 = widen(Xb, "bf16"), widen(Wb, "bf16")
    phi = sls.feature_map(to_torch_x(Xb, "bf16"), to_torch_x(Wb, "bf16"),
                          torch.from_numpy(b).cuda()).cpu().numpy().astype(np.float64)
    want = O.rff_features(X64, W64, b)
    tol = feature_tolerance(X64, W64, b.astype(np.float64))
    assert np.all(np.abs(phi - want) <= tol)


def test_feature_map_tc_cosine_ranges(sls):
    """The tensor-core epilogue's cosine over a wide range of arguments: rows
    scaled so that theta = x.w + b runs from about 1e-3 to beyond 8192 (where
    a 32-column block falls back to the library cosine), and rows of zeros
    (theta = b exactly).  Every feature within the float32 bound of the
    oracle's Eq. rff_map."""
    g = np.random.default_rng(7)
    N, d, D = 384, 64, 512
    X = g.standard_normal((N, d)) / math.sqrt(d)
    scale = np.repeat([1e-3, 1.0, 30.0, 400.0, 20000.0, 0.0], N // 6)
    X = X * scale[:, None]
    Xb = WL.f32_to_bf16_bits(X.astype(np.float32))
    Wb = WL.f32_to_bf16_bits((g.standard_normal((D, d)) * d ** -0.25).astype(np.float32))
    b = (g.random(D) * 2 * math.pi).astype(np.float32)
    X64, W64 = widen(Xb, "bf16"), widen(Wb, "bf16")
    theta = X64 @ W64.T + b.astype(np.float64)
    assert np.max(np.abs(theta)) > 8192.0 and np.min(np.abs(theta)) < 1.0
    phi = sls.feature_map(to_torch_x(Xb, "bf16"), to_torch_x(Wb, "bf16"),
                          torch.from_numpy(b).cuda()).cpu().numpy().astype(np.float64)
    want = O.rff_features(X64, W64, b)
    tol = feature_tolerance(X64, W64, b.astype(np.float64))
    err = np.abs(phi - want)
    assert np.all(err <= tol), float(np.max(err / tol))


def test_feature_map_batched_live_windows(sls):
    """One launch over a batch of prompts (Sec. 3.2) that computes only the
    row tiles touching a live window (Sec. 3.6): computed rows match the
    oracle; tiles with no live window stay unwritten; without flags every row
    of every prompt matches."""
    B, N, rows, d, D, win = 3, 700, 650, 128, 512, 200
    w = WL.scaled(WL.WORKLOADS["mistral7b"], N=N, d=d, D=D)
    prompts = [WL.make_prompt(w, index=k) for k in range(B)]
    prm = WL.make_params(D, d, 8, 8, 1, "bf16")
    Xb = np.stack([pp.X for pp in prompts])
    X = to_torch_x(Xb, "bf16")
    W64 = prm.w_f64()
    tol = [feature_tolerance(pp.x_f64()[:rows], W64, prm.b.astype(np.float64))
           for pp in prompts]
    want = [O.rff_features(pp.x_f64()[:rows], W64, prm.b) for pp in prompts]
    nwin = -(-rows // win)
    live = np.array([[1, 0, 0, 1], [0, 0, 0, 0], [0, 1, 0, 0]], dtype=np.int32)
    assert live.shape == (B, nwin)
    out = torch.full((B * rows, D), float("nan"), device="cuda")
    sls.feature_map_batched(X, to_torch_x(prm.W, "bf16"), torch.from_numpy(prm.b).cuda(), rows,
                            live=torch.from_numpy(live).cuda(), win=win, out=out)
    got = out.cpu().numpy().astype(np.float64).reshape(B, rows, D)
    for k in range(B):
        for t0 in range(0, rows, 128):
            t1 = min(rows, t0 + 128)
            touched = range(t0 // win, (t1 - 1) // win + 1)
            tile = got[k, t0:t1]
            if any(live[k, j] for j in touched):
                assert np.all(np.abs(tile - want[k][t0:t1]) <= tol[k][t0:t1]), (k, t0)
            else:
                assert np.all(np.isnan(tile)), (k, t0)
    full = sls.feature_map_batched(X, to_torch_x(prm.W, "bf16"), torch.from_numpy(prm.b).cuda(),
                                   rows).cpu().numpy().astype(np.float64).reshape(B, rows, D)
    for k in range(B):
        assert np.all(np.abs(full[k] - want[k]) <= tol[k]), k


# ---------------------------------------------------------------------------
# Lanczos + Ritz pairs (Algorithm 2, Algorithm 1)
# ---------------------------------------------------------------------------


def _lanczos_case(sls, phi32, q1, r):
    theta, U, r_eff, alpha, beta = sls.lanczos_topr(torch.from_numpy(phi32).cuda(),
                                                    torch.from_numpy(q1).cuda(), r)
    torch.cuda.synchronize()
    a, b_, Q, k = O.lanczos(phi32.astype(np.float64), q1, r)
    th_o, S_o, U_o = O.ritz_pairs(a, b_, Q)
    k_gpu = int(r_eff.item())
    assert k_gpu == k
    th = theta.cpu().numpy()[:k]
    # Ritz values at the operator's noise floor (|theta| <= 1e-12 theta_1, the
    # null space reached at a breakdown) are zero in exact arithmetic; they are
    # compared against that absolute floor instead of relatively.
    floor = ZERO_FLOOR * abs(th_o[0])
    err = np.abs(th - th_o)
    assert np.all(err <= RITZ_RTOL * np.abs(th_o) + floor), float(np.max(err / (np.abs(th_o) + floor)))
    Ug = U.cpu().numpy()[:, :k]
    assert max_subspace_angle(Ug, U_o) <= ANGLE_TOL
    assert np.all(U.cpu().numpy()[:, k:] == 0.0)
    return th, th_o, Ug, U_o, alpha.cpu().numpy()[:k], a


@pytest.mark.parametrize("name,N,D,r", [("tiny", 500, 256, 16), ("mistral7b", 8180, 1024, 32)])
def test_lanczos_matches_oracle(sls, name, N, D, r):
    w, p, prm = _workload_inputs(name, N=N, D=D)
    phi32 = oracle_phi32(p.x_f64(), prm.w_f64(), prm.b)
    th, th_o, Ug, U_o, al, al_o = _lanczos_case(sls, phi32, prm.q1[:N], r)
    # the diagonal of T entry by entry: each alpha_j carries rounding at the
    # scale of the dominant eigenvalue (every step's matvec holds its
    # component), so the absolute term is a small multiple of max|alpha|
    # times the double-float unit (measured: 3e-9 relative at alpha_7 of
    # the mistral7b shape, max|alpha| = 7952, with the Ritz values at 1e-13)
    assert np.allclose(al, al_o, rtol=1e-9, atol=1e-11 * abs(al_o).max())
    # individual Ritz vectors agree (up to the sign convention, which both
    # sides fix) where the Ritz value is well separated
    gaps = np.minimum(np.abs(np.diff(np.r_[np.inf, th_o])), np.abs(np.diff(np.r_[th_o, -np.inf])))
    for j in range(len(th_o)):
        if gaps[j] > 1e-3 * th_o[0]:
            cosv = float(Ug[:, j] @ U_o[:, j] / np.linalg.norm(Ug[:, j]) / np.linalg.norm(U_o[:, j]))
            assert cosv > 1 - 1e-6, (j, cosv)


@pytest.mark.parametrize("name,N,D,r", [("mistral7b", 3000, 1024, 128),   # KT = 4 (r = SLS_MAX_R)
                                        ("tiny", 2000, 4096, 32),        # GPT = 4
                                        ("tiny", 1500, 8192, 16),        # GPT = 8 (D = SLS_MAX_D)
                                        ("tiny", 333, 8192, 128)])       # both, ragged strips
def test_lanczos_widest_shapes(sls, name, N, D, r):
    """The kernel instantiations for the widest feature counts and the
    largest Krylov rank the interface accepts."""
    w, p, prm = _workload_inputs(name, N=N, D=D)
    phi32 = oracle_phi32(p.x_f64(), prm.w_f64(), prm.b)
    _lanczos_case(sls, phi32, prm.q1[:N], r)


def test_compress_at_interface_limits(sls):
    """The whole pass at D = 8192, r = 128 and b = 32 (the interface's
    maxima): the output invariants and the oracle's macro embeddings and
    positions of the GPU's own groups."""
    w, p, prm = _workload_inputs("tiny", N=900, D=8192)
    prm32 = WL.make_params(8192, w.d, 128, 32, w.N, w.dtype)
    cfg = sls.Config.make(rho=4.0, D=8192, r=128, bits=32, preserve_last=12)
    X = to_torch_x(p.X, w.dtype)
    Xt, pos, t2m, r_eff, _ = sls.compress(
        X, cfg, to_torch_x(prm32.W, w.dtype), torch.from_numpy(prm32.b).cuda(),
        torch.from_numpy(prm32.R).cuda(), torch.from_numpy(prm32.q1).cuda())
    torch.cuda.synchronize()
    M = sls.output_count(cfg, w.N)
    assert int(r_eff[0].item()) == 128
    _check_pass(sls, p.x_f64(), Xt.cpu().numpy(), pos.cpu().numpy(), t2m.cpu().numpy(), M, 0, 12)


def test_lanczos_breakdown_low_rank(sls):
    w, p, prm = _workload_inputs("tiny", N=64, D=64)
    phi = oracle_phi32(p.x_f64()[:5], prm.w_f64()[:64], prm.b[:64])
    g = np.random.default_rng(1)
    phi32 = phi[g.integers(0, 5, size=300)]
    _lanczos_case(sls, phi32, g.standard_normal(300), 16)


def test_lanczos_tiny_sizes(sls):
    g = np.random.default_rng(2)
    for N, D, r in [(1, 4, 4), (3, 8, 8), (40, 12, 16), (257, 20, 7)]:
        X = g.standard_normal((N, 6)) / math.sqrt(6)
        W = g.standard_normal((D, 6)) * 6 ** -0.25
        b = g.random(D) * 2 * math.pi
        phi32 = O.rff_features(X, W, b).astype(np.float32)
        _lanczos_case(sls, phi32, g.standard_normal(N), r)


@pytest.mark.parametrize("N,D,r,distinct", [(2, 4, 4, 2), (5, 64, 16, 5), (16, 256, 16, 16),
                                             (16, 256, 16, 9), (17, 100, 32, 17),
                                             (32, 1024, 32, 20), (32, 256, 8, 32)])
def test_lanczos_window_sizes(sls, N, D, r, distinct):
    """Window-sized problems (N <= 32, the local backend's windows) take the
    warp-per-problem kernel: r_eff (breakdown on repeated tokens), Ritz
    values and subspace against the oracle."""
    g = np.random.default_rng(N * 1000 + D + distinct)
    d = 48
    X = g.standard_normal((distinct, d)) / math.sqrt(d)
    X = X[np.concatenate([np.arange(distinct), g.integers(0, distinct, N - distinct)])]
    W = g.standard_normal((D, d)) * d ** -0.25
    b = g.random(D) * 2 * math.pi
    phi32 = O.rff_features(X, W, b).astype(np.float32)
    _lanczos_case(sls, phi32, g.standard_normal(N), r)


# ---------------------------------------------------------------------------
# SimHash (Sec. 3.3) -- bit-exact given the oracle's U
# ---------------------------------------------------------------------------


def test_simhash_bit_exact_on_oracle_ritz_vectors(sls):
    w, p, prm = _workload_inputs("tiny")
    X = p.x_f64()[:500]
    phi = O.rff_features(X, prm.w_f64(), prm.b)
    a, b_, Q, k = O.lanczos(phi, prm.q1[:500], w.r)
    _, _, U = O.ritz_pairs(a, b_, Q)
    U32 = U.astype(np.float32)
    want = O.simhash(U32, prm.R[:w.bits, :k])
    got = sls.simhash(torch.from_numpy(U32).cuda(), torch.from_numpy(prm.R).cuda(), w.bits)
    assert np.array_equal(got.cpu().numpy().view(np.uint32), want)


@pytest.mark.parametrize("bits,k", [(1, 3), (12, 32), (32, 64), (16, 5)])
def test_simhash_bit_exact_adversarial(sls, bits, k):
    g = np.random.default_rng(bits * 100 + k)
    N = 4099
    U = g.standard_normal((N, k)).astype(np.float32)
    # rows with tiny dot products, exact zeros and negative zeros
    U[:50] *= 1e-30
    U[50:60] = 0.0
    U[60:70] = -0.0
    R = g.standard_normal((bits, k)).astype(np.float32)
    R[0, :] = np.float32(1e-3) * R[0, :]
    want = O.simhash(U, R)
    got = sls.simhash(torch.from_numpy(U).cuda(), torch.from_numpy(R).cuda(), bits)
    assert np.array_equal(got.cpu().numpy().view(np.uint32), want)
    # k taken from a device scalar (r_eff): columns past it are ignored
    kd = torch.tensor([max(1, k - 2)], dtype=torch.int32, device="cuda")
    got2 = sls.simhash(torch.from_numpy(U).cuda(), torch.from_numpy(R).cuda(), bits, k_dev=kd)
    want2 = O.simhash(U[:, :max(1, k - 2)], R)
    assert np.array_equal(got2.cpu().numpy().view(np.uint32), want2)


# ---------------------------------------------------------------------------
# clusters, adjustment, positions and macro-tokens (Sec. 3.3-3.4)
# ---------------------------------------------------------------------------


def _oracle_aggregate(X64, codes, M, scheme, renorm):
    clusters = O.bucket(codes)
    groups = O.adjust_groups(clusters, M)
    order = O.order_groups(groups, scheme)
    Xt = O.aggregate_groups(X64, [groups[i] for i in order], renorm)
    pos = np.array([O.group_position(groups[i], scheme) for i in order])
    t2m = np.empty(len(codes), dtype=np.int64)
    for k, i in enumerate(order):
        t2m[groups[i]] = k
    return Xt, pos, t2m, len(clusters)


@pytest.mark.parametrize("scheme", [O.POS_MAX, O.POS_MEDIAN, O.POS_MEAN])
@pytest.mark.parametrize("case", ["merge", "split", "equal"])
def test_aggregate_bit_exact_maps(sls, scheme, case):
    g = np.random.default_rng(7 + scheme)
    N, d = 3001, 64
    X = (g.standard_normal((N, d)) / 8).astype(np.float32)
    nb = {"merge": 900, "split": 40, "equal": 300}[case]
    codes = g.integers(0, nb, size=N).astype(np.uint32) * np.uint32(2654435761 % 2 ** 32 // 7)
    C = len(set(codes.tolist()))
    M = {"merge": max(1, C // 3), "split": min(N, C * 7 + 3), "equal": C}[case]
    Xt_o, pos_o, t2m_o, C_o = _oracle_aggregate(X.astype(np.float64), codes, M, scheme, True)
    Xt, pos, t2m = sls.aggregate(torch.from_numpy(X).cuda(),
                                 torch.from_numpy(codes.view(np.int32)).cuda(), M, scheme, True)
    assert np.array_equal(t2m.cpu().numpy(), t2m_o)
    assert np.array_equal(pos.cpu().numpy(), pos_o)
    assert np.max(np.abs(Xt.cpu().numpy() - Xt_o)) <= EMB_TOL


@pytest.mark.parametrize("scheme", [O.POS_MAX, O.POS_MEDIAN, O.POS_MEAN])
@pytest.mark.parametrize("case", ["merge", "split", "equal"])
def test_aggregate_bit_exact_maps_one_large_problem(sls, scheme, case):
    """A single problem large enough for the grid-wide segment kernel."""
    g = np.random.default_rng(11 + scheme)
    N, d = 20000, 16
    X = (g.standard_normal((N, d)) / 4).astype(np.float32)
    nb = {"merge": 6000, "split": 130, "equal": 2000}[case]
    codes = g.integers(0, nb, size=N).astype(np.uint32) * np.uint32(2654435761 % 2 ** 32 // 7)
    C = len(set(codes.tolist()))
    M = {"merge": max(1, C // 3), "split": min(N, C * 7 + 3), "equal": C}[case]
    Xt_o, pos_o, t2m_o, C_o = _oracle_aggregate(X.astype(np.float64), codes, M, scheme, True)
    Xt, pos, t2m = sls.aggregate(torch.from_numpy(X).cuda(),
                                 torch.from_numpy(codes.view(np.int32)).cuda(), M, scheme, True)
    assert np.array_equal(t2m.cpu().numpy(), t2m_o)
    assert np.array_equal(pos.cpu().numpy(), pos_o)
    assert np.max(np.abs(Xt.cpu().numpy() - Xt_o)) <= EMB_TOL


@pytest.mark.parametrize("scheme", [O.POS_MAX, O.POS_MEDIAN, O.POS_MEAN])
@pytest.mark.parametrize("N", [1, 2, 5, 16, 17, 31, 32])
def test_aggregate_window_sized_bit_exact(sls, scheme, N):
    """Problems of at most 32 tokens (the local backend's windows) take the
    one-warp segment kernel: merge, split (D'Hondt, repeated sizes and ties)
    and equal cases against the oracle, bit-exact maps and positions."""
    g = np.random.default_rng(100 * N + scheme)
    d = 24
    X = (g.standard_normal((N, d)) / 5).astype(np.float32)
    for nb in (1, 2, 3, max(1, N // 2), N):
        codes = (g.integers(0, nb, size=N).astype(np.uint32) * np.uint32(40503)) ^ np.uint32(7)
        C = len(set(codes.tolist()))
        for M in sorted({1, max(1, C - 1), C, min(N, C + 1), min(N, 2 * C + 1), N}):
            Xt_o, pos_o, t2m_o, _ = _oracle_aggregate(X.astype(np.float64), codes, M, scheme,
                                                      True)
            Xt, pos, t2m = sls.aggregate(torch.from_numpy(X).cuda(),
                                         torch.from_numpy(codes.view(np.int32)).cuda(), M,
                                         scheme, True)
            assert np.array_equal(t2m.cpu().numpy(), t2m_o), (nb, M)
            assert np.array_equal(pos.cpu().numpy(), pos_o), (nb, M)
            assert np.max(np.abs(Xt.cpu().numpy() - Xt_o)) <= EMB_TOL


def test_aggregate_bf16_large_groups(sls):
    """bf16 embeddings, duplicated tokens (one large cluster), renorm off and on."""
    w, p, prm = _workload_inputs("mistral7b", N=6000, d=512)
    X64 = p.x_f64()
    g = np.random.default_rng(3)
    codes = (p.ids % 700).astype(np.uint32)
    codes[g.random(6000) < 0.3] = 5  # a cluster holding ~30% of the tokens
    for renorm, M in [(True, 375), (False, 375), (True, 1500)]:
        Xt_o, pos_o, t2m_o, _ = _oracle_aggregate(X64, codes, M, O.POS_MAX, renorm)
        Xt, pos, t2m = sls.aggregate(to_torch_x(p.X, "bf16"),
                                     torch.from_numpy(codes.view(np.int32)).cuda(), M,
                                     O.POS_MAX, renorm)
        assert np.array_equal(t2m.cpu().numpy(), t2m_o)
        assert np.array_equal(pos.cpu().numpy(), pos_o)
        assert np.max(np.abs(Xt.cpu().numpy() - Xt_o)) <= EMB_TOL


def test_aggregate_edge_cases(sls):
    g = np.random.default_rng(4)
    X = (g.standard_normal((17, 8)) / 3).astype(np.float32)
    for codes, M in [(np.zeros(17, np.uint32), 1), (np.zeros(17, np.uint32), 17),
                     (np.arange(17, dtype=np.uint32), 17), (np.arange(17, dtype=np.uint32), 1),
                     (np.full(17, 0xFFFFFFFF, np.uint32), 5)]:
        Xt_o, pos_o, t2m_o, _ = _oracle_aggregate(X.astype(np.float64), codes, M, O.POS_MAX, True)
        Xt, pos, t2m = sls.aggregate(torch.from_numpy(X).cuda(),
                                     torch.from_numpy(codes.view(np.int32)).cuda(), M)
        assert np.array_equal(t2m.cpu().numpy(), t2m_o)
        assert np.array_equal(pos.cpu().numpy(), pos_o)
        assert np.max(np.abs(Xt.cpu().numpy() - Xt_o)) <= EMB_TOL


# ---------------------------------------------------------------------------
# whole pass (Algorithm 1, backends of Sec. 3.5 and 3.6)
# ---------------------------------------------------------------------------


def _check_pass(sls, X64, Xt, pos, t2m, M, pf, pl, scheme=O.POS_MAX, renorm=True):
    """Invariants of the output, and the macro embeddings / positions the
    oracle computes from the GPU's own token map."""
    N = X64.shape[0]
    t2m = t2m.astype(np.int64)
    assert t2m.min() >= 0 and t2m.max() == M - 1
    assert np.all(np.bincount(t2m, minlength=M) >= 1)
    for i in range(pf):
        assert t2m[i] == i and pos[i] == i
    for i in range(pl):
        assert t2m[N - pl + i] == M - pl + i and pos[M - pl + i] == N - pl + i
    groups = [np.nonzero(t2m == m)[0] for m in range(M)]
    Xt_o = O.aggregate_groups(X64, groups, renorm)
    assert np.max(np.abs(Xt - Xt_o)) <= EMB_TOL
    pos_o = np.array([O.group_position(gm, scheme) for gm in groups])
    assert np.array_equal(pos, pos_o)
    if scheme == O.POS_MAX:
        assert np.all(np.diff(pos) > 0)


def test_compress_global_tiny(sls):
    w, p, prm = _workload_inputs("tiny")
    cfg = sls.Config.make(rho=w.rho, D=w.D, r=w.r, bits=w.bits, preserve_last=12)
    X = to_torch_x(p.X, w.dtype)
    Xt, pos, t2m, r_eff, route = sls.compress(
        X, cfg, to_torch_x(prm.W, w.dtype), torch.from_numpy(prm.b).cuda(),
        torch.from_numpy(prm.R).cuda(), torch.from_numpy(prm.q1).cuda())
    M = sls.output_count(cfg, w.N)
    assert M == O.target_count(w.N - 12, w.rho) + 12
    _check_pass(sls, p.x_f64(), Xt.cpu().numpy(), pos.cpu().numpy(), t2m.cpu().numpy(), M, 0, 12)
    assert int(r_eff[0].item()) == w.r
    # the oracle's own run: same cluster-count regime (diagnostic agreement)
    ocfg = O.CompressConfig(rho=w.rho, D=w.D, r=w.r, bits=w.bits)
    res = O.compress_global(p.x_f64(), prm.w_f64(), prm.b, prm.R, prm.q1, ocfg)
    assert res.Xt.shape[0] == M


def test_compress_global_batched(sls):
    """The global backend on a batch of prompts of equal length: one Lanczos
    problem per prompt in one launch of the batched plan.  Per prompt: r_eff
    against the oracle, the output invariants and the oracle's macro
    embeddings and positions of the GPU's own groups."""
    w = WL.scaled(WL.WORKLOADS["mistral7b"], N=900, d=64, D=256, r=16, bits=10, rho=4.0)
    prompts = [WL.make_prompt(w, index=i) for i in range(3)]
    prm = WL.make_params(256, 64, 16, 32, 3 * 900, "bf16")
    X = to_torch_x(np.stack([pp.X for pp in prompts]), "bf16")
    cfg = sls.Config.make(rho=4.0, D=256, r=16, bits=10, preserve_first=2, preserve_last=12)
    Xt, pos, t2m, r_eff, _ = sls.compress(X, cfg, to_torch_x(prm.W, "bf16"),
                                          torch.from_numpy(prm.b).cuda(),
                                          torch.from_numpy(prm.R).cuda(),
                                          torch.from_numpy(prm.q1).cuda())
    torch.cuda.synchronize()
    M = sls.output_count(cfg, 900)
    for i, pp in enumerate(prompts):
        res = O.compress_global(pp.x_f64(), prm.w_f64(), prm.b, prm.R,
                                prm.q1[i * 900:(i + 1) * 900],
                                O.CompressConfig(rho=4.0, D=256, r=16, bits=10, preserve_first=2,
                                                 preserve_last=12))
        assert int(r_eff[i].item()) == res.info["r_eff"]
        _check_pass(sls, pp.x_f64(), Xt[i].cpu().numpy(), pos[i].cpu().numpy(),
                    t2m[i].cpu().numpy(), M, 2, 12)


@pytest.mark.parametrize("scheme,mode,pf,pl", [(O.POS_MEDIAN, 0, 3, 5), (O.POS_MEAN, 0, 0, 0),
                                               (O.POS_MAX, 1, 2, 12)])
def test_compress_options(sls, scheme, mode, pf, pl):
    w, p, prm = _workload_inputs("tiny")
    cfg = sls.Config.make(rho=3.0, D=64, r=8, bits=6, preserve_first=pf, preserve_last=pl,
                          pos_scheme=scheme, pos_mode=mode)
    X = to_torch_x(p.X, w.dtype)
    Xt, pos, t2m, _, _ = sls.compress(X, cfg, to_torch_x(prm.W[:64], w.dtype),
                                      torch.from_numpy(prm.b[:64]).cuda(),
                                      torch.from_numpy(prm.R).cuda(),
                                      torch.from_numpy(prm.q1).cuda())
    M = sls.output_count(cfg, w.N)
    t2m = t2m.cpu().numpy()
    pos = pos.cpu().numpy()
    if mode == 1:
        assert np.array_equal(pos, np.arange(M))
    else:
        _check_pass(sls, p.x_f64(), Xt.cpu().numpy(), pos, t2m, M, pf, pl, scheme)


def test_compress_identity_and_degenerate(sls):
    w, p, prm = _workload_inputs("tiny")
    X = to_torch_x(p.X, w.dtype)
    for rho in (1.0, 0.5):
        cfg = sls.Config.make(rho=rho)
        Xt, pos, t2m, _, _ = sls.compress(X, cfg)
        assert torch.equal(Xt, X.float())
        assert np.array_equal(pos.cpu().numpy(), np.arange(w.N))
        assert np.array_equal(t2m.cpu().numpy(), np.arange(w.N))
    cfg = sls.Config.make(rho=4.0, preserve_last=w.N + 3)
    Xt, pos, t2m, _, _ = sls.compress(X, cfg)
    assert torch.equal(Xt, X.float())
    # all tokens identical: one cluster, split into M pieces.  Phi has rank 1,
    # so the Krylov space is span{q1, A q1} and Lanczos stops after 2 steps.
    Xs = X[:1].repeat(100, 1).contiguous()
    cfg = sls.Config.make(rho=4.0, D=64, r=8, bits=4, preserve_last=0)
    Xt, pos, t2m, r_eff, _ = sls.compress(Xs, cfg, to_torch_x(prm.W[:64], w.dtype),
                                          torch.from_numpy(prm.b[:64]).cuda(),
                                          torch.from_numpy(prm.R).cuda(),
                                          torch.from_numpy(prm.q1).cuda())
    assert int(r_eff[0].item()) == 2
    _check_pass(sls, Xs.double().cpu().numpy(), Xt.cpu().numpy(), pos.cpu().numpy(),
                t2m.cpu().numpy(), 25, 0, 0)


def test_compress_chunk_backend(sls):
    w, p, prm = _workload_inputs("tiny")
    X = to_torch_x(p.X, w.dtype)
    cfg = sls.Config.make(backend=sls.BACKEND_CHUNK, rho=4.0, preserve_last=12)
    Xt, pos, t2m, _, _ = sls.compress(X, cfg)
    res = O.compress_chunk(p.x_f64(), O.CompressConfig(rho=4.0, preserve_last=12))
    assert np.array_equal(t2m.cpu().numpy(), res.tok2macro)
    assert np.array_equal(pos.cpu().numpy(), res.pos)
    assert np.max(np.abs(Xt.cpu().numpy() - res.Xt)) <= EMB_TOL


@pytest.mark.parametrize("D", [64, 256])
def test_compress_adaptive_small_batch(sls, D):
    """Adaptive router on a batch of 3 prompts (windows of 96): route flags,
    budgets and chunk windows against the oracle; spectral windows by their
    invariants.  D = 256 takes the batched tensor-core feature map, whose
    128-row tiles straddle the windows."""
    w = WL.scaled(WL.WORKLOADS["adaptive"], N=700, d=64, batch=3)
    prompts = [WL.make_prompt(w, index=i, dup_frac=WL.adaptive_dup_frac(i, 3)) for i in range(3)]
    prm = WL.make_params(D, 64, 8, 32, 3 * 700, "bf16")
    Xb = np.stack([pp.X for pp in prompts])
    X = to_torch_x(Xb, "bf16")
    for rho in (2.0, 4.0, 16.0):
        cfg = sls.Config.make(backend=sls.BACKEND_ADAPTIVE, rho=rho, D=D, r=8, window=96,
                              preserve_last=12)
        Xt, pos, t2m, r_eff, route = sls.compress(X, cfg, to_torch_x(prm.W, "bf16"),
                                                  torch.from_numpy(prm.b).cuda(),
                                                  torch.from_numpy(prm.R).cuda(),
                                                  torch.from_numpy(prm.q1).cuda())
        M = sls.output_count(cfg, 700)
        nw = len(O.window_bounds(688, 96))
        route = route.cpu().numpy()[:3 * nw].reshape(3, nw)
        for i, pp in enumerate(prompts):
            ocfg = O.CompressConfig(rho=rho, D=D, r=8, window=96, preserve_last=12)
            res = O.compress_adaptive(pp.x_f64(), prm.w_f64(), prm.b, prm.R,
                                      prm.q1[i * 700:(i + 1) * 700], ocfg)
            tau = O.tau_schedule(rho)
            for k, (sp, sc) in enumerate(zip(res.info["spectral"], res.info["scores"])):
                if rho >= 16 or abs(sc - tau) > 1e-5:
                    assert route[i, k] == int(sp), (rho, i, k, sc)
            _check_pass(sls, pp.x_f64(), Xt[i].cpu().numpy(), pos[i].cpu().numpy(),
                        t2m[i].cpu().numpy(), M, 0, 12)
            # every macro-token lies inside one window
            t = t2m[i].cpu().numpy()
            for m in range(M - 12):
                mem = np.nonzero(t == m)[0]
                assert mem.min() // 96 == mem.max() // 96
            # chunk windows match the oracle exactly
            bounds = O.window_bounds(688, 96)
            for k, (s, e) in enumerate(bounds):
                if not route[i, k]:
                    assert np.array_equal(t[s:e], res.tok2macro[s:e])


def _planted_adaptive_batch():
    """Two low-redundancy prompts with a few windows made redundant (three
    rows repeated over the window), so that the router sends those windows
    to the spectral path and the rest to the chunk path."""
    w = WL.scaled(WL.WORKLOADS["adaptive"], N=1000, d=64, batch=2)
    X = np.stack([WL.make_prompt(w, index=i, dup_frac=0.0).X for i in range(2)]).copy()
    for (i, k) in [(0, 1), (0, 4), (1, 2)]:
        s0 = k * 96
        X[i, s0:s0 + 96] = np.resize(X[i, s0:s0 + 3], (96, 64))
    prm = WL.make_params(256, 64, 8, 32, 2 * 1000, "bf16")
    return X, prm


def _adaptive_case(sls, X, prm, rho, pl, scheme=O.POS_MAX, mode=0, renorm=1):
    B = X.shape[0]
    cfg = sls.Config.make(backend=sls.BACKEND_ADAPTIVE, rho=rho, D=256, r=8, window=96,
                          preserve_last=pl, pos_scheme=scheme, pos_mode=mode, renorm=renorm)
    Xt, pos, t2m, r_eff, route = sls.compress(to_torch_x(X, "bf16"), cfg,
                                              to_torch_x(prm.W, "bf16"),
                                              torch.from_numpy(prm.b).cuda(),
                                              torch.from_numpy(prm.R).cuda(),
                                              torch.from_numpy(prm.q1).cuda())
    torch.cuda.synchronize()
    M = sls.output_count(cfg, 1000)
    bounds = O.window_bounds(1000 - pl, 96)
    route = route.cpu().numpy()[:B * len(bounds)].reshape(B, len(bounds))
    routes = []
    for i in range(B):
        x64 = WL.bf16_bits_to_f32(X[i]).astype(np.float64)
        res = O.compress_adaptive(x64, prm.w_f64(), prm.b, prm.R, prm.q1[i * 1000:(i + 1) * 1000],
                                  O.CompressConfig(rho=rho, D=256, r=8, window=96,
                                                   preserve_last=pl, pos_scheme=scheme,
                                                   pos_mode=mode, renorm=bool(renorm)))
        tau = O.tau_schedule(rho)
        for k, (sp, sc) in enumerate(zip(res.info["spectral"], res.info["scores"])):
            if abs(sc - tau) > 1e-5:
                assert route[i, k] == int(sp), (rho, i, k, sc)
        if mode == O.MODE_COMPACT:
            assert np.array_equal(pos[i].cpu().numpy(), np.arange(M))
        else:
            _check_pass(sls, x64, Xt[i].cpu().numpy(), pos[i].cpu().numpy(),
                        t2m[i].cpu().numpy(), M, 0, pl, scheme, bool(renorm))
        t = t2m[i].cpu().numpy()
        for k, (s_, e_) in enumerate(bounds):
            if not route[i, k]:  # chunk windows: the oracle's output exactly
                assert np.array_equal(t[s_:e_], res.tok2macro[s_:e_])
                ms = np.unique(res.tok2macro[s_:e_])
                assert np.array_equal(pos[i].cpu().numpy()[ms], res.pos[ms])
                assert np.max(np.abs(Xt[i].cpu().numpy()[ms] - res.Xt[ms])) <= EMB_TOL
        routes.append(route[i])
    return np.array(routes)


def test_compress_adaptive_mixed_routes(sls):
    """Below rho = 16 the score pass writes every window's chunk output and
    the spectral windows replace theirs: a batch with both kinds of window."""
    X, prm = _planted_adaptive_batch()
    for rho in (2.0, 4.0, 8.0):
        routes = _adaptive_case(sls, X, prm, rho, 12)
        assert routes.sum() >= 1 and (routes == 0).sum() >= 1


@pytest.mark.parametrize("scheme,mode,renorm", [(O.POS_MEDIAN, 0, 1), (O.POS_MEAN, 0, 0),
                                                (O.POS_MAX, 1, 1)])
def test_compress_adaptive_options(sls, scheme, mode, renorm):
    """The score pass's chunk outputs under the other position schemes, the
    compact position mode and without the renormalisation."""
    X, prm = _planted_adaptive_batch()
    routes = _adaptive_case(sls, X, prm, 4.0, 12, scheme, mode, renorm)
    assert (routes == 0).sum() >= 1


def test_compress_adaptive_all_chunk_no_preserved(sls):
    """Every window on the chunk path and no preserved tokens: the
    aggregation has no work item at all."""
    X, prm = _planted_adaptive_batch()
    routes = _adaptive_case(sls, X[:1], prm, 2.0, 0)
    assert routes.sum() == 0


BREAK_BAND = 30.0


def _reff_agrees(phi, q1, r, tol, r_gpu):
    """r_eff of Algorithm 2 on one window against the oracle.  Equal, or one
    apart where the oracle's beta_j / max_i(|alpha_i| + beta_i) at the step in
    question lies within a factor BREAK_BAND of tol: there beta is rounding
    noise amplified near a breakdown (Phi of lower rank than r), the decision
    belongs to the rounding, and both outcomes are Algorithm 2 executed
    exactly up to rounding (the factor is the ratio of the double-float and
    float64 unit roundoffs of the two matvecs)."""
    a, be, _, _ = O.lanczos(phi, q1, r, tol=0.0)
    rel = be / np.maximum.accumulate(np.abs(a[:len(be)]) + be)
    hit = np.nonzero(rel <= tol)[0]
    r_o = int(hit[0]) + 1 if hit.size else len(a)
    if r_gpu == r_o:
        return True
    if abs(r_gpu - r_o) != 1:
        return False
    j = min(r_gpu, r_o) - 1
    return tol / BREAK_BAND <= rel[j] <= tol * BREAK_BAND


@pytest.mark.parametrize("dtype,D", [("bf16", 256), ("f32", 64)])
def test_compress_local_w16(sls, dtype, D):
    """Local LSH at the paper's default window of 16 (Sec. 3.5): every window
    spectral with its exact budget; r_eff per window matches the oracle; at
    rho = 16 every window is one macro-token, so the whole output matches the
    oracle; otherwise the invariants and the per-window macro counts."""
    w = WL.scaled(WL.WORKLOADS["mistral7b"], N=700, d=64, D=D, dtype=dtype)
    p = WL.make_prompt(w)
    prm = WL.make_params(D, 64, 16, 16, 700, dtype)
    X = to_torch_x(p.X, dtype)
    X64 = p.x_f64()
    Nc = 688
    bounds = O.window_bounds(Nc, 16)
    for rho in (2.0, 4.0, 16.0):
        cfg = sls.Config.make(backend=sls.BACKEND_LOCAL, rho=rho, D=D, r=16, window=16,
                              preserve_last=12)
        Xt, pos, t2m, r_eff, route = sls.compress(X, cfg, to_torch_x(prm.W, dtype),
                                                  torch.from_numpy(prm.b).cuda(),
                                                  torch.from_numpy(prm.R).cuda(),
                                                  torch.from_numpy(prm.q1).cuda())
        M = sls.output_count(cfg, 700)
        ocfg = O.CompressConfig(rho=rho, D=D, r=16, window=16, preserve_last=12)
        res = O.compress_local(X64, prm.w_f64(), prm.b, prm.R, prm.q1, ocfg)
        assert np.all(route.cpu().numpy()[:len(bounds)] == 1)
        rg = r_eff.cpu().numpy()[:len(bounds)]
        for k, (s_, e_) in enumerate(bounds):
            if rg[k] != res.info["r_eff"][k]:
                phi = oracle_phi32(X64[s_:e_], prm.w_f64(), prm.b).astype(np.float64)
                assert _reff_agrees(phi, prm.q1[s_:e_], 16, 1e-10, int(rg[k])), (rho, k)
        assert np.mean(rg == np.array(res.info["r_eff"])) >= 0.9
        t = t2m.cpu().numpy()
        _check_pass(sls, X64, Xt.cpu().numpy(), pos.cpu().numpy(), t, M, 0, 12)
        for (s_, e_), m in zip(bounds, res.info["budgets"]):
            assert len(np.unique(t[s_:e_])) == m
        if rho >= 16:
            assert np.array_equal(t, res.tok2macro)
            assert np.array_equal(pos.cpu().numpy(), res.pos)
            assert np.max(np.abs(Xt.cpu().numpy() - res.Xt)) <= EMB_TOL


# ---------------------------------------------------------------------------
# row-normalised operator (Sec. 3.2 variant)
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("name,N,D", [("tiny", 500, 256), ("mistral7b", 3000, 1024),
                                      ("tiny", 777, 2048), ("tiny", 130, 8192), ("tiny", 97, 4)])
def test_feature_normalize_matches_oracle(sls, name, N, D):
    """Rows scaled by 1/sqrt(s_i), s = Phi (Phi^T 1): s to the float64
    rounding level, every scaled element within one float32 ulp of the
    oracle's float64 value rounded to float32."""
    w, p, prm = _workload_inputs(name, N=N, D=D)
    phi32 = oracle_phi32(p.x_f64(), prm.w_f64(), prm.b)
    s_o, phin_o = O.normalized_features(phi32.astype(np.float64))
    t = torch.from_numpy(phi32).cuda()
    s = sls.feature_normalize(t).cpu().numpy()
    assert np.allclose(s, s_o, rtol=1e-12, atol=0)
    got = t.cpu().numpy()
    want = phin_o.astype(np.float32)
    ulp = np.spacing(np.abs(want).astype(np.float32))
    assert np.all(np.abs(got - want) <= ulp)


def test_lanczos_normalized_operator(sls):
    """Lanczos on the GPU's normalised rows against the oracle on the same
    float32 rows; the top Ritz value of the normalised operator is 1."""
    w, p, prm = _workload_inputs("mistral7b", N=3000, D=1024)
    phi32 = oracle_phi32(p.x_f64(), prm.w_f64(), prm.b)
    t = torch.from_numpy(phi32).cuda()
    sls.feature_normalize(t)
    phin = t.cpu().numpy()
    th, th_o, Ug, U_o, _, _ = _lanczos_case(sls, phin, prm.q1[:3000], 32)
    assert abs(th[0] - 1.0) < 1e-5 and abs(th_o[0] - 1.0) < 1e-5


@pytest.mark.parametrize("backend", ["global", "local"])
def test_compress_normalized(sls, backend):
    w, p, prm = _workload_inputs("tiny")
    kw = dict(rho=w.rho, D=w.D, r=w.r, bits=w.bits, preserve_last=12, normalize=1)
    if backend == "local":
        cfg = sls.Config.make(backend=sls.BACKEND_LOCAL, window=16, **kw)
    else:
        cfg = sls.Config.make(**kw)
    X = to_torch_x(p.X, w.dtype)
    Xt, pos, t2m, r_eff, route = sls.compress(
        X, cfg, to_torch_x(prm.W, w.dtype), torch.from_numpy(prm.b).cuda(),
        torch.from_numpy(prm.R).cuda(), torch.from_numpy(prm.q1).cuda())
    M = sls.output_count(cfg, w.N)
    _check_pass(sls, p.x_f64(), Xt.cpu().numpy(), pos.cpu().numpy(), t2m.cpu().numpy(), M, 0, 12)
    if backend == "global":
        assert int(r_eff[0].item()) == w.r

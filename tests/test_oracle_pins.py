"""Pins for the CPU oracle (no GPU): each check ties an oracle function to
something other than itself -- closed forms, library routines, dense
eigendecompositions, statistics the paper states, invariants, brute force on
tiny inputs and values printed in the paper (tests/golden/paper_values.json)."""
import json
import math
import os

import numpy as np
import pytest
import scipy.linalg

import oracle as O
import workloads as WL

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _tiny_inputs(N=64, d=16, D=128, seed=3):
    g = np.random.default_rng(seed)
    X = g.standard_normal((N, d)) / math.sqrt(d)
    W = g.standard_normal((D, d)) * d ** -0.25
    b = g.random(D) * 2 * math.pi
    return X, W, b


# ---------------------------------------------------------------------------
# RFF map (Sec. 3.2, Eq. rff_map and Eq. bochner)
# ---------------------------------------------------------------------------


def test_rff_expectation_is_gaussian_kernel():
    """E[phi(x)^T phi(y)] = exp(-|x-y|^2 / (2 sqrt d)) when Omega has variance
    1/sqrt(d): pins the variance reading, the sqrt(2/D) scale and the phase b."""
    N, d, D = 24, 16, 1 << 16
    g = np.random.default_rng(11)
    X = g.standard_normal((N, d)) / math.sqrt(d) * 1.5
    W = g.standard_normal((D, d)) * d ** -0.25
    b = g.random(D) * 2 * math.pi
    Phi = O.rff_features(X, W, b)
    K = Phi @ Phi.T
    sq = ((X[:, None, :] - X[None, :, :]) ** 2).sum(-1)
    Kg = np.exp(-sq / (2 * math.sqrt(d)))
    assert np.max(np.abs(K - Kg)) < 0.03
    # the unnormalised softmax kernel exp(x^T y / sqrt d) up to the diagonal
    # scaling exp(|x|^2 / 2 sqrt d) (Sec. 3.2)
    kappa = np.exp(X @ X.T / math.sqrt(d))
    s = np.exp((X ** 2).sum(1) / (2 * math.sqrt(d)))
    assert np.max(np.abs(K * s[:, None] * s[None, :] - kappa) / kappa) < 0.05
    # a wrong variance (1/d) would give a visibly different kernel
    Kwrong = np.exp(-sq / (2 * d))
    assert np.max(np.abs(Kwrong - Kg)) > 0.1


def test_rff_shape_and_bounds():
    X, W, b = _tiny_inputs()
    Phi = O.rff_features(X, W, b)
    assert Phi.shape == (64, 128)
    assert np.all(np.abs(Phi) <= math.sqrt(2 / 128) + 1e-15)


# ---------------------------------------------------------------------------
# Lanczos (Algorithm 2) and Ritz pairs (Algorithm 1)
# ---------------------------------------------------------------------------


def _phi(N=300, d=24, D=64, seed=5):
    X, W, b = _tiny_inputs(N, d, D, seed)
    return O.rff_features(X, W, b)


def test_lanczos_full_rank_reproduces_dense_spectrum():
    Phi = _phi()
    N, D = Phi.shape
    q1 = np.random.default_rng(1).standard_normal(N)
    alpha, beta, Q, r_eff = O.lanczos(Phi, q1, D + 1)
    theta, S, U = O.ritz_pairs(alpha, beta, Q)
    lam = np.sort(np.linalg.eigvalsh(Phi @ Phi.T))[::-1]   # dense N x N
    k = min(40, D)
    assert np.allclose(theta[:k], lam[:k], rtol=1e-10, atol=1e-10 * lam[0])


def test_gram_spectrum_equals_dense():
    Phi = _phi()
    lam_dense = np.sort(np.linalg.eigvalsh(Phi @ Phi.T))[::-1][:Phi.shape[1]]
    lam_gram = np.sort(np.linalg.eigvalsh(Phi.T @ Phi))[::-1]
    assert np.allclose(lam_dense, lam_gram, rtol=1e-9, atol=1e-9 * lam_gram[0])


def test_lanczos_interlacing_orthonormality_and_projection():
    Phi = _phi(N=400, D=96)
    N = Phi.shape[0]
    q1 = np.random.default_rng(2).standard_normal(N)
    r = 16
    alpha, beta, Q, r_eff = O.lanczos(Phi, q1, r)
    assert r_eff == r
    theta, S, U = O.ritz_pairs(alpha, beta, Q)
    lam = np.sort(np.linalg.eigvalsh(Phi.T @ Phi))[::-1]
    # Cauchy interlacing / Thm 2 upper bound: theta_j <= lambda_j
    assert np.all(theta <= lam[:r] * (1 + 1e-12) + 1e-12)
    # top Ritz value converged to the dominant eigenvalue
    assert abs(theta[0] - lam[0]) / lam[0] < 1e-10
    # Q^T Q = I and T = Q^T A Q
    assert np.max(np.abs(Q.T @ Q - np.eye(r))) < 1e-12
    A = Phi @ Phi.T
    T = np.diag(alpha) + np.diag(beta, 1) + np.diag(beta, -1)
    assert np.max(np.abs(Q.T @ A @ Q - T)) < 1e-10 * lam[0]
    # eigenpairs of T
    assert np.allclose(T @ S, S * theta[None, :], atol=1e-10 * lam[0])
    assert np.all(S[0] > 0)
    assert np.all(np.diff(theta) <= 0)


def test_lanczos_breakdown_on_low_rank():
    """Phi with k distinct rows has rank <= k, so the Krylov space has
    dimension <= k + 1 and Algorithm 2 must stop early."""
    base = _phi(N=5, D=64)
    g = np.random.default_rng(3)
    Phi = base[g.integers(0, 5, size=200)]
    q1 = g.standard_normal(200)
    alpha, beta, Q, r_eff = O.lanczos(Phi, q1, 16)
    assert 1 <= r_eff <= 6
    assert alpha.size == r_eff and beta.size == r_eff - 1
    assert np.max(np.abs(Q.T @ Q - np.eye(r_eff))) < 1e-10


def test_ritz_values_match_gram_on_tiny_workload():
    w = WL.WORKLOADS["tiny"]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()[:500]
    Phi = O.rff_features(X, prm.w_f64(), prm.b)
    alpha, beta, Q, r_eff = O.lanczos(Phi, prm.q1[:500], w.r)
    theta, S, U = O.ritz_pairs(alpha, beta, Q)
    lam = np.sort(np.linalg.eigvalsh(Phi.T @ Phi))[::-1]
    # residual certificate |A u - theta u| = beta_r |S[r-1, j]| for converged pairs
    A = Phi @ Phi.T
    res = np.linalg.norm(A @ U - U * theta[None, :], axis=0)
    for j in range(4):
        assert abs(theta[j] - lam[j]) <= res[j] + 1e-9 * lam[0]
    # the dominant eigenvalue carries most of the energy (K2 kill test, Sec. 5.5)
    assert theta[0] > 0.5 * X.shape[0]


# ---------------------------------------------------------------------------
# SimHash (Sec. 3.3, Eq. simhash, Eq. lsh_collision)
# ---------------------------------------------------------------------------


def test_simhash_brute_force_scalar_float32():
    g = np.random.default_rng(4)
    U = g.standard_normal((7, 5)).astype(np.float32)
    R = g.standard_normal((6, 5)).astype(np.float32)
    codes = O.simhash(U, R)
    for i in range(7):
        code = 0
        for l in range(6):
            acc = np.float32(0.0)
            for m in range(5):
                acc = np.float32(acc + np.float32(U[i, m] * R[l, m]))
            if acc > np.float32(0.0):
                code |= 1 << l
        assert int(codes[i]) == code


def test_simhash_bit_order_and_zero():
    U = np.array([[1.0, 0.0], [-1.0, 0.0], [0.0, 1.0], [0.0, 0.0], [-0.0, -0.0]],
                 dtype=np.float32)
    R = np.array([[1.0, 0.0], [-1.0, 0.0], [0.0, 1.0]], dtype=np.float32)
    codes = O.simhash(U, R)
    assert codes.tolist() == [0b001, 0b010, 0b100, 0, 0]


def test_simhash_collision_probability():
    """Per-bit collision rate -> 1 - angle/pi (Eq. lsh_collision, b = 1), and
    all-b-bit collisions -> (1 - angle/pi)^b."""
    g = np.random.default_rng(9)
    k = 8
    x = g.standard_normal(k)
    y = g.standard_normal(k)
    ang = math.acos(x @ y / np.linalg.norm(x) / np.linalg.norm(y))
    p1 = 1 - ang / math.pi
    n = 32 * 1600
    R = g.standard_normal((n, k)).astype(np.float32)
    U = np.stack([x, y]).astype(np.float32)
    same = 0
    for t in range(n // 32):
        c = O.simhash(U, R[32 * t:32 * t + 32])
        same += 32 - bin(int(c[0]) ^ int(c[1])).count("1")
    rate = same / n
    assert abs(rate - p1) < 4 * math.sqrt(p1 * (1 - p1) / n)
    # through the oracle, 4-bit codes from independent hyperplane blocks
    b = 4
    trials = 8000
    hits = 0
    for t in range(trials):
        Rt = R[(t * b) % (n - b):(t * b) % (n - b) + b]
        c = O.simhash(U, Rt)
        hits += int(c[0] == c[1])
    pb = p1 ** b
    assert abs(hits / trials - pb) < 4 * math.sqrt(pb * (1 - pb) / trials)


def test_auto_bits_and_target_count():
    assert O.auto_bits(4096, 4.0) == 10 and O.auto_bits(4097, 4.0) == 11
    assert O.auto_bits(1, 4.0) == 1
    assert O.target_count(16372, 8.0) == 2047
    assert O.target_count(16372, 16.0) == 1024


def test_golden_actual_rho_table4():
    """Table 4's actual ratios are reproduced by N=16384 with the last 12
    tokens preserved and M* = ceil(N_c / rho) (not round)."""
    g = _golden()["actual_rho"]
    N, pl = g["N"], g["preserve_last"]
    for rho, actual in g["cases"]:
        M = O.target_count(N - pl, rho) + pl
        assert round(N / M, 3) == actual
    # the round-to-nearest reading fails the 16x case
    M_round = round((N - pl) / 16.0) + pl
    assert round(N / M_round, 3) != 15.815


def test_golden_complexity():
    g = _golden()["complexity"]
    per = O.complexity_ops(g["d"], g["D"], g["r"], g["b"])
    assert abs(per - g["ops_per_token_approx"]) / g["ops_per_token_approx"] < g["rel_tol_per_token"]
    tot = per * g["N"]
    assert abs(tot - g["ops_total_approx"]) / g["ops_total_approx"] < g["rel_tol_total"]


# ---------------------------------------------------------------------------
# Buckets and the exact-length adjustment (Sec. 3.3)
# ---------------------------------------------------------------------------


def test_bucket_partition_and_order():
    g = np.random.default_rng(5)
    codes = g.integers(0, 9, size=200).astype(np.uint32)
    cl = O.bucket(codes)
    allm = np.concatenate(cl)
    assert sorted(allm.tolist()) == list(range(200))
    cc = [int(codes[c[0]]) for c in cl]
    assert cc == sorted(set(codes.tolist()))
    for c in cl:
        assert np.all(np.diff(c) > 0) and np.all(codes[c] == codes[c[0]])


def test_array_split_sizes_match_numpy():
    for n in range(1, 30):
        for p in range(1, n + 1):
            assert O.array_split_sizes(n, p) == [len(a) for a in np.array_split(np.arange(n), p)]


def _dhondt_invariant(sizes, seats):
    """Highest-averages property: every extra seat awarded has a quotient at
    least as large as any seat not awarded."""
    awarded = [sizes[c] / seats[c] for c in range(len(sizes)) if seats[c] >= 2]
    unawarded = [sizes[c] / (seats[c] + 1) for c in range(len(sizes)) if seats[c] < sizes[c]]
    if awarded and unawarded:
        assert min(awarded) >= max(unawarded) - 1e-12


def test_dhondt_textbook_and_invariants():
    # votes 100/80/30/20 with 8 seats: plain D'Hondt gives 4/3/1/0; with one
    # guaranteed seat per cluster the last cluster is seated and the remaining
    # four seats go to the quotients 50, 40, 33.3, 26.7 -> 3/3/1/1.
    assert O.dhondt_seats([100, 80, 30, 20], 8) == [3, 3, 1, 1]
    # with 12 seats plain D'Hondt already seats everyone (6/4/1/1); the
    # variant must agree, including the tie at quotient 20 (A and B both seated).
    assert O.dhondt_seats([100, 80, 30, 20], 12) == [6, 4, 1, 1]
    g = np.random.default_rng(6)
    for t in range(200):
        C = int(g.integers(1, 12))
        sizes = g.integers(1, 40, size=C).tolist()
        M = int(g.integers(C, sum(sizes) + 1))
        seats = O.dhondt_seats(sizes, M)
        assert sum(seats) == M
        assert all(1 <= p <= n for p, n in zip(seats, sizes))
        _dhondt_invariant(sizes, seats)


def test_dhondt_brute_force_tiny():
    """Among all allocations with 1 <= p_c <= n_c summing to M, the D'Hondt
    seats maximise the smallest quotient n_c / p_c over clusters holding an
    extra seat, and among ties take seats from the later clusters first."""
    import itertools
    g = np.random.default_rng(8)
    for t in range(60):
        C = int(g.integers(1, 5))
        sizes = g.integers(1, 7, size=C).tolist()
        M = int(g.integers(C, sum(sizes) + 1))
        best = None
        for alloc in itertools.product(*[range(1, n + 1) for n in sizes]):
            if sum(alloc) != M:
                continue
            ok = True
            for c in range(C):
                for c2 in range(C):
                    if alloc[c] >= 2 and alloc[c2] < sizes[c2]:
                        lhs = sizes[c] * (alloc[c2] + 1)
                        rhs = sizes[c2] * alloc[c]
                        if lhs < rhs or (lhs == rhs and c2 < c):
                            ok = False
            if ok:
                assert best is None, (sizes, M)
                best = list(alloc)
        assert best == O.dhondt_seats(sizes, M), (sizes, M)


def test_adjust_merge_and_split():
    g = np.random.default_rng(7)
    codes = g.integers(0, 50, size=300).astype(np.uint32)
    cl = O.bucket(codes)
    C = len(cl)
    for M in [1, 5, C - 1, C, C + 1, C + 30, 300]:
        groups = O.adjust_groups(cl, M)
        assert len(groups) == M
        assert sorted(np.concatenate(groups).tolist()) == list(range(300))
        assert all(len(x) >= 1 for x in groups)
        if M < C:
            # each group is a union of clusters of consecutive code rank
            rank = {int(codes[c[0]]): t for t, c in enumerate(cl)}
            for x in groups:
                ranks = sorted({rank[int(codes[i])] for i in x})
                assert ranks == list(range(ranks[0], ranks[-1] + 1))
        if M > C:
            # each group is a contiguous piece (in index order) of one cluster
            for x in groups:
                assert len({int(codes[i]) for i in x}) == 1
                c = cl[[int(codes[cc[0]]) for cc in cl].index(int(codes[x[0]]))]
                pos = np.searchsorted(c, x)
                assert np.all(np.diff(pos) == 1)


# ---------------------------------------------------------------------------
# Aggregation and positions (Sec. 3.4)
# ---------------------------------------------------------------------------


def test_group_position_matches_library():
    g = np.random.default_rng(9)
    for t in range(100):
        m = g.choice(1000, size=int(g.integers(1, 20)), replace=False)
        assert O.group_position(m, O.POS_MAX) == int(np.max(m))
        if m.size % 2 == 1:
            assert O.group_position(m, O.POS_MEDIAN) == int(np.median(m))
        else:
            assert O.group_position(m, O.POS_MEDIAN) == int(np.sort(m)[m.size // 2 - 1])
        mean = float(np.mean(m))
        assert O.group_position(m, O.POS_MEAN) == int(math.floor(mean + 0.5))


def test_aggregate_invariants():
    g = np.random.default_rng(10)
    X = g.standard_normal((50, 8))
    groups = [np.array([0]), np.array([1, 2, 3]), np.arange(4, 50)]
    out = O.aggregate_groups(X, groups, renorm=True)
    assert np.array_equal(out[0], X[0])
    for k in (1, 2):
        eta = np.linalg.norm(X[groups[k]], axis=1).mean()
        assert abs(np.linalg.norm(out[k]) - eta) < 1e-12 * eta
        cosv = out[k] @ X[groups[k]].mean(0) / np.linalg.norm(out[k]) / np.linalg.norm(X[groups[k]].mean(0))
        assert cosv > 1 - 1e-12
    plain = O.aggregate_groups(X, groups, renorm=False)
    assert np.allclose(plain[2], np.mean(X[4:50], axis=0), atol=1e-15)
    same = np.tile(X[:1], (5, 1))
    assert np.allclose(O.aggregate_groups(same, [np.arange(5)])[0], X[0], atol=1e-15)


def _check_result(res, N, M_expected, pf, pl, scheme=O.POS_MAX):
    M = res.Xt.shape[0]
    assert M == M_expected
    assert res.tok2macro.min() >= 0 and res.tok2macro.max() == M - 1
    counts = np.bincount(res.tok2macro, minlength=M)
    assert np.all(counts >= 1) and counts.sum() == N
    for i in range(pf):
        assert res.tok2macro[i] == i and res.pos[i] == i
    for i in range(pl):
        assert res.tok2macro[N - pl + i] == M - pl + i and res.pos[M - pl + i] == N - pl + i
    if scheme == O.POS_MAX:
        assert np.all(np.diff(res.pos) > 0)     # K1 kill test: monotone positions
        for m in range(M):
            assert res.pos[m] == np.max(np.nonzero(res.tok2macro == m)[0])


def test_compress_global_tiny_invariants():
    w = WL.WORKLOADS["tiny"]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    cfg = O.CompressConfig(rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                           preserve_last=w.preserve_last)
    res = O.compress_global(p.x_f64(), prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
    Nc = w.N - w.preserve_last
    _check_result(res, w.N, O.target_count(Nc, w.rho) + w.preserve_last, 0, 12)
    X = p.x_f64()
    # each macro-token has the mean member norm
    for m in range(res.Xt.shape[0]):
        mem = np.nonzero(res.tok2macro == m)[0]
        eta = np.linalg.norm(X[mem], axis=1).mean()
        assert abs(np.linalg.norm(res.Xt[m]) - eta) < 1e-12 * max(eta, 1)
    assert res.info["r_eff"] == w.r


def test_compress_identity_bypass():
    w = WL.WORKLOADS["tiny"]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()
    for rho in (1.0, 0.5):
        cfg = O.CompressConfig(rho=rho, D=w.D, r=w.r)
        res = O.compress_global(X, prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
        assert np.array_equal(res.Xt, X)
        assert np.array_equal(res.pos, np.arange(w.N))
    cfg = O.CompressConfig(rho=4.0, preserve_last=w.N + 5)
    res = O.compress_global(X, prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
    assert np.array_equal(res.Xt, X)


def test_compress_position_modes_and_schemes():
    w = WL.WORKLOADS["tiny"]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()[:200]
    for scheme in (O.POS_MEDIAN, O.POS_MEAN):
        cfg = O.CompressConfig(rho=4.0, D=64, r=8, bits=6, pos_scheme=scheme,
                               preserve_first=3, preserve_last=5)
        res = O.compress_global(X, prm.w_f64()[:64], prm.b[:64], prm.R, prm.q1, cfg)
        _check_result(res, 200, O.target_count(192, 4.0) + 8, 3, 5, scheme)
        assert np.all(np.diff(res.pos) >= 0)
    cfg = O.CompressConfig(rho=4.0, D=64, r=8, bits=6, pos_mode=O.MODE_COMPACT)
    res = O.compress_global(X, prm.w_f64()[:64], prm.b[:64], prm.R, prm.q1, cfg)
    assert np.array_equal(res.pos, np.arange(res.Xt.shape[0]))


def test_compress_chunk_closed_form():
    g = np.random.default_rng(12)
    X = g.standard_normal((37, 6))
    cfg = O.CompressConfig(rho=4.0, preserve_last=5, renorm=False)
    res = O.compress_chunk(X, cfg)
    # groups of 4 over the first 32 tokens, then 5 preserved
    assert res.Xt.shape[0] == 8 + 5
    for k in range(8):
        assert np.allclose(res.Xt[k], X[4 * k:4 * k + 4].mean(0), atol=1e-15)
        assert res.pos[k] == 4 * k + 3


# ---------------------------------------------------------------------------
# Adaptive router (Sec. 3.6)
# ---------------------------------------------------------------------------


def test_tau_schedule_golden():
    for rho, tau in _golden()["tau_schedule"]["points"]:
        assert abs(O.tau_schedule(rho) - tau) < 1e-12
    assert abs(O.tau_schedule(4.0) - 0.65) < 1e-12
    assert O.tau_schedule(64.0) == 0.55 and O.tau_schedule(1.5) == 0.70


def test_redundancy_score_closed_forms():
    g = np.random.default_rng(13)
    x = g.standard_normal(16)
    assert abs(O.redundancy_score(np.tile(x, (9, 1))) - 1.0) < 1e-12
    L = 10
    E = np.eye(16)[:L]
    assert abs(O.redundancy_score(E) - 1 / math.sqrt(L)) < 1e-12
    Z = np.vstack([E, np.zeros((2, 16))])
    # zero rows contribute 0 but count in L
    assert abs(O.redundancy_score(Z) - (L / math.sqrt(L)) / (L + 2)) < 1e-12
    assert O.redundancy_score(np.vstack([x, -x])) == 0.0


def test_window_budgets():
    g = np.random.default_rng(14)
    for t in range(200):
        Nc = int(g.integers(1, 5000))
        w = int(g.integers(1, 600))
        lens = [e - s for s, e in O.window_bounds(Nc, w)]
        assert sum(lens) == Nc and all(0 < L <= w for L in lens)
        rho = float(g.choice([1.5, 2, 4, 8, 16]))
        M = O.target_count(Nc, rho)
        if M < len(lens):
            continue
        bud = O.window_budgets(lens, M)
        assert sum(bud) == M
        assert all(1 <= m <= L for m, L in zip(bud, lens))
        # proportional: full windows differ by at most one
        full = [m for m, L in zip(bud, lens) if L == w]
        if full:
            assert max(full) - min(full) <= 1


def test_route_rules_and_adaptive_invariants():
    w = WL.scaled(WL.WORKLOADS["tiny"], N=512)
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()
    for rho in (2.0, 4.0, 16.0):
        cfg = O.CompressConfig(rho=rho, D=64, r=8, window=96, preserve_last=12)
        res = O.compress_adaptive(X, prm.w_f64()[:64], prm.b[:64], prm.R,
                                  prm.q1, cfg)
        Nc = 500
        _check_result(res, 512, O.target_count(Nc, rho) + 12, 0, 12)
        bounds = O.window_bounds(Nc, 96)
        sp = res.info["spectral"]
        if rho >= 16:
            assert all(sp)
        for (s, e), f, sc in zip(bounds, sp, res.info["scores"]):
            if rho < 16 and e - s <= 4:
                assert not f
            if rho < 16 and e - s > 4:
                assert f == (sc >= O.tau_schedule(rho))
        # every macro-token lies inside one window (causal safety of windows)
        for m in range(res.Xt.shape[0] - 12):
            mem = np.nonzero(res.tok2macro == m)[0]
            assert mem.min() // 96 == mem.max() // 96
    # tiny last window is routed to chunk
    spf, _ = O.route_windows(X[:100], [(0, 96), (96, 100)], 4.0, O.CompressConfig())
    assert spf[1] is False


def test_local_backend_reductions():
    """Local LSH (Sec. 3.5) against what fixes it: at rho >= 16 the adaptive
    backend is local LSH (Sec. 3.6); one window over the whole region is the
    global backend; a budget of one macro-token per window makes every window
    one group, i.e. the chunk backend with k = window."""
    w = WL.scaled(WL.WORKLOADS["tiny"], N=300)
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()
    W64, b, R, q1 = prm.w_f64()[:64], prm.b[:64], prm.R, prm.q1

    def same(a, c):
        return (np.array_equal(a.tok2macro, c.tok2macro) and np.array_equal(a.pos, c.pos)
                and np.array_equal(a.Xt, c.Xt))

    cfg = O.CompressConfig(rho=16.0, D=64, r=8, window=40, preserve_last=12)
    assert same(O.compress_local(X, W64, b, R, q1, cfg),
                O.compress_adaptive(X, W64, b, R, q1, cfg))
    cfg = O.CompressConfig(rho=4.0, D=64, r=8, window=1000, preserve_last=12)
    assert same(O.compress_local(X, W64, b, R, q1, cfg),
                O.compress_global(X, W64, b, R, q1, cfg))
    cfg = O.CompressConfig(rho=16.0, D=64, r=8, window=16, preserve_last=12)
    res = O.compress_local(X, W64, b, R, q1, cfg)
    assert same(res, O.compress_chunk(X, cfg))
    assert all(res.info["spectral"])


def test_local_backend_w16_invariants():
    """w = 16 (the paper's default): every window yields exactly its budget
    of macro-tokens, none crosses a window, positions are causal."""
    w = WL.scaled(WL.WORKLOADS["tiny"], N=500)
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X = p.x_f64()
    for rho in (2.0, 4.0, 8.0):
        cfg = O.CompressConfig(rho=rho, D=64, r=16, window=16, preserve_last=12)
        res = O.compress_local(X, prm.w_f64()[:64], prm.b[:64], prm.R, prm.q1, cfg)
        Nc = 488
        _check_result(res, 500, O.target_count(Nc, rho) + 12, 0, 12)
        bounds = O.window_bounds(Nc, 16)
        budgets = res.info["budgets"]
        assert sum(budgets) == O.target_count(Nc, rho)
        t = res.tok2macro[:Nc]
        for (s_, e_), m in zip(bounds, budgets):
            assert len(np.unique(t[s_:e_])) == m
        for m in range(res.Xt.shape[0] - 12):
            mem = np.nonzero(res.tok2macro == m)[0]
            assert mem.min() // 16 == mem.max() // 16
        assert all(1 <= k <= 16 for k in res.info["r_eff"])


def test_normalized_operator_pins():
    """The row-normalised operator (Sec. 3.2 variant) against what fixes it:
    D^{-1/2} K D^{-1/2} with D = diag(K 1) has eigenvalue exactly 1 with
    eigenvector D^{1/2} 1 (K (1) = D 1), its largest for a kernel with positive
    entries; its spectrum is that of diag(s)^-1 K (similar matrices); Lanczos
    on the scaled rows finds theta_1 = 1; positive row scales leave SimHash
    codes unchanged."""
    w = WL.scaled(WL.WORKLOADS["tiny"], N=200)
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    Phi = O.rff_features(p.x_f64(), prm.w_f64(), prm.b)
    K = Phi @ Phi.T
    s, Phin = O.normalized_features(Phi)
    assert np.allclose(s, K.sum(axis=1), rtol=1e-12)
    assert np.all(K > 0) and np.all(s > 0)
    S = Phin @ Phin.T
    assert np.allclose(S, K / np.sqrt(np.outer(s, s)), rtol=1e-11, atol=0)
    ev, V = np.linalg.eigh(S)
    assert abs(ev[-1] - 1.0) < 1e-12
    u = np.sqrt(s) / np.linalg.norm(np.sqrt(s))
    assert abs(abs(V[:, -1] @ u) - 1.0) < 1e-10
    evP = np.sort(np.linalg.eigvals(K / s[:, None]).real)
    assert np.allclose(evP, np.sort(ev), atol=1e-11)
    a, be, Q, k = O.lanczos(Phin, prm.q1[:200], 16)
    th, S_, U = O.ritz_pairs(a, be, Q)
    assert abs(th[0] - 1.0) < 1e-10
    g = np.random.default_rng(3)
    U32 = U.astype(np.float32)
    scale = (g.random(U.shape[0]) + 0.5).astype(np.float32)
    R = prm.R[:8, :k]
    assert np.array_equal(O.simhash(U32, R), O.simhash(U32 * scale[:, None], R))


def test_normalized_compress_invariants():
    w = WL.WORKLOADS["tiny"]
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    cfg = O.CompressConfig(rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                           preserve_last=w.preserve_last, normalize=True)
    res = O.compress_global(p.x_f64(), prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
    _check_result(res, w.N, O.target_count(w.N - 12, w.rho) + 12, 0, 12)
    assert abs(res.info["theta"][0] - 1.0) < 1e-6


# ---------------------------------------------------------------------------
# input embeddings (Sec. 3.1, Fig. 1): X = E[ids]
# ---------------------------------------------------------------------------


def test_embed_lookup_is_the_one_hot_product():
    """The lookup equals the product of the one-hot token matrix with the
    table (a row of zeros for an id with no row), element for element."""
    rng = np.random.default_rng(5)
    V, d = 37, 9
    table = rng.standard_normal((V, d))
    ids = rng.integers(-3, V + 3, size=400)
    onehot = (ids[:, None] == np.arange(V)[None, :]).astype(np.float64)
    X = O.embed_lookup(table, ids)
    assert X.shape == (400, d) and X.dtype == table.dtype
    assert np.array_equal(X, onehot @ table)
    assert np.all(X[(ids < 0) | (ids >= V)] == 0)


def test_embed_lookup_reproduces_the_prompt_generator():
    """The seeded prompts are table lookups: the bf16 table of every vocabulary
    row, looked up at the prompt's ids, is the prompt's X bit for bit (so a
    device-resident table and the ids stand in for X)."""
    w = WL.scaled(WL.WORKLOADS["qwen7b"], N=300, d=32, V=400)
    p = WL.make_prompt(w)
    table = WL.f32_to_bf16_bits(
        WL.vocab_rows(WL.DATA_SEED, np.arange(w.V), w.d).astype(np.float32))
    X = O.embed_lookup(table, p.ids)
    assert X.dtype == np.uint16 and np.array_equal(X, p.X)


# ---------------------------------------------------------------------------
# bfloat16 storage of the feature matrix (opt-in half-size Phi)
# ---------------------------------------------------------------------------


def test_bf16_round_closed_forms():
    """Representable values stay; halfway cases go to the even neighbour; the
    spacing below 2^-126 is 2^-133; signs and zeros are kept."""
    r = O.bf16_round
    for v in [1.0, 1.5, -3.0, 2.0 ** -100, 2.0 ** 100, 1 + 2.0 ** -7, 0.0]:
        assert r(np.array([v]))[0] == v
    assert r(np.array([1 + 2.0 ** -8]))[0] == 1.0                  # tie -> even (1.0)
    assert r(np.array([1 + 3 * 2.0 ** -8]))[0] == 1 + 2.0 ** -6    # tie -> even (k = 2)
    assert r(np.array([1 + 2.0 ** -8 + 2.0 ** -30]))[0] == 1 + 2.0 ** -7  # above the tie
    assert r(np.array([-(1 + 3 * 2.0 ** -8)]))[0] == -(1 + 2.0 ** -6)
    assert r(np.array([2.0 ** -133 * 2.5]))[0] == 2.0 ** -132      # subnormal tie -> even
    assert np.signbit(r(np.array([-0.0]))[0])


def test_bf16_round_matches_bit_level_rounding():
    """Against the input generator's independent bit-level rounding of
    float32 values (round-to-nearest-even on the high 16 bits), over many
    magnitudes, and within half a unit of the 8-bit significand."""
    rng = np.random.default_rng(11)
    x = (rng.standard_normal(200000) * np.exp2(rng.integers(-60, 60, 200000))).astype(np.float32)
    want = WL.bf16_bits_to_f32(WL.f32_to_bf16_bits(x)).astype(np.float64)
    got = O.bf16_round(x.astype(np.float64))
    assert np.array_equal(got, want)
    assert np.all(np.abs(got - x) <= 2.0 ** -8 * np.abs(x))


def test_bf16_storage_tolerance_class():
    """The opt-in bf16 Phi defines a nearby operator: its eigenvalues are
    within ||Phi_b Phi_b^T - Phi Phi^T||_2 <= (2 u + u^2) ||Phi||_2^2
    (u = 2^-8, bf16's unit roundoff) of the float32 ones (Weyl), and the Lanczos run on it keeps
    the leading Ritz value within that bound -- far below the RFF estimate's
    own error O(D^-1/2) -- while the Ritz subspace moves measurably (which
    is why bf16 storage is opt-in with its own tolerance class)."""
    w = WL.scaled(WL.WORKLOADS["tiny"], N=400)
    p, prm = WL.make_prompt(w), WL.params_for(w)
    phi = O.rff_features(p.x_f64(), prm.w_f64(), prm.b).astype(np.float32).astype(np.float64)
    phib = O.bf16_round(phi)
    u = 2.0 ** -8
    assert np.all(np.abs(phib - phi) <= u * np.abs(phi))
    lam = np.linalg.eigvalsh(phi @ phi.T)
    lamb = np.linalg.eigvalsh(phib @ phib.T)
    bound = (2 * u + u * u) * np.linalg.norm(phi, 2) ** 2
    assert np.max(np.abs(lam - lamb)) <= bound
    a, b_, Q, k = O.lanczos(phi, prm.q1[:w.N], w.r)
    ab, bb, Qb, kb = O.lanczos(phib, prm.q1[:w.N], w.r)
    th = O.ritz_pairs(a, b_, Q)[0]
    thb = O.ritz_pairs(ab, bb, Qb)[0]
    assert abs(th[0] - thb[0]) <= bound
    assert bound < th[0] / math.sqrt(w.D)

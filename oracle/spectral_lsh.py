"""Spectral-LSH, stated step by step in numpy (test infrastructure only).

Citations are to the paper's sections, equations and algorithms:
  Eq. rff_map / Eq. implicit_matvec   -- Sec. 3.2
  Algorithm 1 (pipeline), Algorithm 2 (implicit Lanczos)
  Eq. simhash, target count b = ceil(log2(N/rho)), adjust step -- Sec. 3.3
  Eq. macro_embed, position schemes   -- Sec. 3.4
  Backends, preservation              -- Sec. 3.5
  Eq. redundancy, routing, budgets    -- Sec. 3.6 and App. B.3 / B.8
  Identity bypass for rho <= 1        -- Sec. 5.6 and App. B.6
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np
import scipy.linalg

__all__ = [
    "CompressConfig", "rff_features", "lanczos", "ritz_pairs", "simhash",
    "auto_bits", "target_count", "bucket", "dhondt_seats", "adjust_groups",
    "array_split_sizes", "group_position", "aggregate_groups", "order_groups",
    "compress_global", "tau_schedule", "redundancy_score", "window_bounds",
    "window_budgets", "route_windows", "chunk_groups", "spectral_groups",
    "compress_adaptive", "compress_local", "compress_chunk", "complexity_ops",
    "CompressResult",
    "POS_MAX", "POS_MEDIAN", "POS_MEAN", "MODE_REPRESENTATIVE", "MODE_COMPACT",
    "normalized_features", "embed_lookup", "bf16_round",
]

# ---------------------------------------------------------------------------
# Configuration (mirrors the paper's CompressionConfig, App. B.3 and B.8)
# ---------------------------------------------------------------------------

POS_MAX, POS_MEDIAN, POS_MEAN = 0, 1, 2
MODE_REPRESENTATIVE, MODE_COMPACT = 0, 1


@dataclasses.dataclass
class CompressConfig:
    rho: float = 4.0
    D: int = 256
    r: int = 16
    bits: int = 0                 # 0 = ceil(log2(N_c / rho)), Sec. 3.3
    preserve_first: int = 0       # App. B.3
    preserve_last: int = 12       # App. B.3
    pos_scheme: int = POS_MAX     # Sec. 3.4, default max
    pos_mode: int = MODE_REPRESENTATIVE  # Sec. 5.6 / App. B.3
    renorm: bool = True           # Eq. macro_embed
    lanczos_tol: float = 1e-10    # break threshold of Algorithm 2 (reading)
    window: int = 2048            # adaptive / local backend window
    normalize: bool = False       # row-normalised operator (Sec. 3.2 variant)
    tau: float = 0.70             # fixed threshold (App. B.3)
    tau_schedule: bool = True     # compression-aware schedule (Sec. 3.6)


@dataclasses.dataclass
class CompressResult:
    Xt: np.ndarray        # (M, d) float64 macro-token embeddings
    pos: np.ndarray       # (M,) int64 positions
    tok2macro: np.ndarray  # (N,) int64 macro index of every token
    info: dict


# ---------------------------------------------------------------------------
# Step 0: input embeddings (Sec. 3.1, Fig. 1)
# ---------------------------------------------------------------------------


def embed_lookup(table: np.ndarray, ids: np.ndarray) -> np.ndarray:
    """The prompt's input embeddings: row ids[i] of the model's input
    embedding table for token i (Sec. 3.1 takes X from the LLM's input
    embedding layer; Fig. 1 draws prompt tokens -> input embeddings).

    Values are copied as stored (same dtype as the table).  An id outside
    [0, V) has no row: this statement of the lookup gives it a zero row (the
    paper never feeds one)."""
    table = np.asarray(table)
    ids = np.asarray(ids, dtype=np.int64)
    V = table.shape[0]
    X = np.zeros(ids.shape + table.shape[1:], dtype=table.dtype)
    for i, v in enumerate(ids.reshape(-1)):
        if 0 <= v < V:
            X.reshape(-1, *table.shape[1:])[i] = table[v]
    return X


# ---------------------------------------------------------------------------
# Step 1: random Fourier features (Sec. 3.2, Eq. rff_map)
# ---------------------------------------------------------------------------


def rff_features(X: np.ndarray, W: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Phi = sqrt(2/D) * cos(X Omega + b) with W = Omega^T stored D x d.

    Eq. rff_map writes cos(Omega x + b) with Omega in R^{d x D}; the product
    is read as x^T Omega (the only shape that type-checks), and Omega's
    entries are N(0, 1/sqrt(d)) with 1/sqrt(d) the VARIANCE (as the
    covariance I/d^{1/2} of Sec. 3.2 states).  Computed in float64 from the
    exact input values."""
    X = np.asarray(X, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    D = W.shape[0]
    return math.sqrt(2.0 / D) * np.cos(X @ W.T + b[None, :])


def bf16_round(x: np.ndarray) -> np.ndarray:
    """The feature matrix stored in bfloat16 (the opt-in half-size storage of
    Phi): every value rounded to 8 significant bits, to nearest with ties to
    even, returned as float64.

    Reading: the paper computes Eq. rff_map without fixing a storage
    precision (its runs use float16 throughout, App. B); bf16 keeps float32's
    exponent range, and its relative rounding error (2^-8) is several times below
    the Monte-Carlo error of the RFF estimate itself (O(D^-1/2), Sec. 3.2),
    so the stored features define a slightly different operator on which
    Algorithm 2 then runs exactly.  Domain: finite |x| below the bf16
    maximum; values under 2^-126 keep bf16's subnormal spacing 2^-133."""
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)                       # x = f 2^e, 1/2 <= |f| < 1
    e = np.maximum(e, -125)                  # subnormal range: spacing 2^-133
    scale = np.ldexp(1.0, e - 8)             # spacing of 8-bit significands
    return np.round(x / scale) * scale       # np.round: ties to even


# ---------------------------------------------------------------------------
# Step 2: implicit Lanczos (Algorithm 2, Eq. implicit_matvec)
# ---------------------------------------------------------------------------


def lanczos(Phi: np.ndarray, q1: np.ndarray, r: int, tol: float = 1e-10):
    """Algorithm 2 on the implicit operator A(v) = Phi (Phi^T v).

    Readings where Algorithm 2 is silent:
      * the start vector q1 is an input (N(0,1) draws), normalised here;
      * "full re-orthogonalization" is two passes of classical Gram-Schmidt
        against all previous basis vectors (q_1..q_j);
      * the break test "beta_j < tau" uses tau = tol * max_{i<=j}(|alpha_i| +
        beta_i), a scale-relative threshold;
      * exactly r matvecs are taken; beta_r is computed and unused.

    Returns (alpha[r_eff], beta[r_eff-1], Q[N, r_eff], r_eff)."""
    Phi = np.asarray(Phi, dtype=np.float64)
    N = Phi.shape[0]
    q = np.asarray(q1, dtype=np.float64).copy()
    q /= np.linalg.norm(q)
    r = int(min(r, N)) if N > 0 else 0
    Q = np.zeros((N, max(r, 1)))
    alpha: List[float] = []
    beta: List[float] = []
    q_prev = np.zeros(N)
    b_prev = 0.0
    scale = 0.0
    r_eff = 0
    for j in range(r):
        Q[:, j] = q
        z = Phi @ (Phi.T @ q)                 # implicit matvec, Eq. implicit_matvec
        a = float(q @ z)                      # alpha_j = q_j^T z
        z = z - a * q - b_prev * q_prev       # three-term recurrence
        for _ in range(2):                    # full re-orthogonalisation (CGS2)
            Qj = Q[:, :j + 1]
            z = z - Qj @ (Qj.T @ z)
        b = float(np.linalg.norm(z))          # beta_j
        alpha.append(a)
        r_eff = j + 1
        scale = max(scale, abs(a) + b)
        if j == r - 1 or b <= tol * scale:
            break
        beta.append(b)
        q_prev, q, b_prev = q, z / b, b
    return (np.array(alpha), np.array(beta[:max(r_eff - 1, 0)]),
            Q[:, :r_eff].copy(), r_eff)


def normalized_features(Phi: np.ndarray):
    """The cheap normalised operator of Sec. 3.2, diag(s)^-1 Phi (Phi^T v) with
    row sums s = Phi (Phi^T 1), taken in its symmetric form
    D^{-1/2} Phi Phi^T D^{-1/2} (D = diag(s)): the same eigenvalues (the two
    are similar), eigenvectors D^{1/2}-scaled, which SimHash cannot see (a
    positive row scale keeps every sign).  It is the unnormalised operator of
    the rows Phi_i / sqrt(s_i); a row with s_i <= 0 has no positive mass and is
    scaled by 0.  Returns (s, the scaled rows)."""
    Phi = np.asarray(Phi, dtype=np.float64)
    s = Phi @ Phi.sum(axis=0)
    w = np.zeros_like(s)
    pos = s > 0
    w[pos] = 1.0 / np.sqrt(s[pos])
    return s, Phi * w[:, None]


# ---------------------------------------------------------------------------
# Step 3: Eigh(T) and Ritz vectors (Algorithm 1)
# ---------------------------------------------------------------------------


def ritz_pairs(alpha: np.ndarray, beta: np.ndarray, Q: np.ndarray):
    """lambda, V = Eigh(T); Ritz values in descending order and Ritz vectors
    U = Q V (Algorithm 1, Eigh and the top-k Ritz vectors with k = r_eff,
    Z = V-hat).  Each eigenvector of T is signed so that its first component
    is positive (a convention; the paper leaves the sign free)."""
    k = alpha.size
    if k == 1:
        theta = alpha.copy()
        S = np.ones((1, 1))
    else:
        w, V = scipy.linalg.eigh_tridiagonal(alpha, beta)
        order = np.argsort(-w, kind="stable")
        theta = w[order]
        S = V[:, order]
    sgn = np.where(S[0, :] < 0, -1.0, 1.0)
    S = S * sgn[None, :]
    U = Q @ S
    return theta, S, U


# ---------------------------------------------------------------------------
# Step 4: SimHash in the spectral subspace (Sec. 3.3, Eq. simhash)
# ---------------------------------------------------------------------------


def simhash(U32: np.ndarray, R32: np.ndarray) -> np.ndarray:
    """Codes h_i = sum_l [r_l^T z_i > 0] 2^l (bit l <- hyperplane l).

    The dot products use a fixed float32 chain: acc starts at +0.0f and, for
    m = 0..k-1 in order, acc = fl32(acc + fl32(U[i,m] * R[l,m])) with the
    multiply and the add rounded separately (round to nearest even).  A zero
    (+0 or -0) or NaN dot product gives bit 0.  Uses the first k columns of
    R where k = U.shape[1]."""
    U32 = np.ascontiguousarray(U32, dtype=np.float32)
    R32 = np.ascontiguousarray(R32, dtype=np.float32)
    N, k = U32.shape
    bits = R32.shape[0]
    assert bits <= 32 and R32.shape[1] >= k
    acc = np.zeros((N, bits), dtype=np.float32)
    with np.errstate(over="ignore", invalid="ignore"):
        for m in range(k):
            prod = np.multiply(U32[:, m:m + 1], R32[None, :, m], dtype=np.float32)
            acc = np.add(acc, prod, dtype=np.float32)
    codes = np.zeros(N, dtype=np.uint64)
    for l in range(bits):
        codes |= (acc[:, l] > 0).astype(np.uint64) << np.uint64(l)
    return codes.astype(np.uint32)


def auto_bits(n: int, rho: float) -> int:
    """b = ceil(log2(n / rho)) (Sec. 3.3), the smallest b >= 1 with
    2^b * rho >= n, capped at 32."""
    b = 1
    while b < 32 and (2.0 ** b) * rho < n:
        b += 1
    return b


def target_count(n: int, rho: float) -> int:
    """M* = ceil(n / rho) macro-tokens for n compressible tokens (Sec. 3.3)."""
    return int(math.ceil(n / rho))


# ---------------------------------------------------------------------------
# Step 5: buckets and the exact-length adjustment (Sec. 3.3)
# ---------------------------------------------------------------------------


def bucket(codes: np.ndarray) -> List[np.ndarray]:
    """Tokens with identical codes form a cluster (Algorithm 1).  Clusters are
    returned in ascending code order, members in ascending token index."""
    codes = np.asarray(codes, dtype=np.uint64)
    idx = np.arange(codes.size)
    order = sorted(range(codes.size), key=lambda i: (int(codes[i]), i))
    order = np.array(order, dtype=np.int64)
    clusters: List[np.ndarray] = []
    start = 0
    for s in range(1, codes.size + 1):
        if s == codes.size or codes[order[s]] != codes[order[start]]:
            clusters.append(idx[order[start:s]])
            start = s
    return clusters


def dhondt_seats(sizes: Sequence[int], seats: int) -> List[int]:
    """Seats per cluster by the D'Hondt highest-averages method with one seat
    guaranteed per cluster: every cluster starts with one seat, then each
    further seat goes to the cluster with the largest quotient
    n_c / (s_c + 1); ties go to the cluster that comes first (lower code).
    Quotients are compared exactly as integer cross products."""
    C = len(sizes)
    s = [1] * C
    for _ in range(seats - C):
        best = -1
        for c in range(C):
            if s[c] >= sizes[c]:
                continue
            if best < 0 or sizes[c] * (s[best] + 1) > sizes[best] * (s[c] + 1):
                best = c
        s[best] += 1
    return s


def array_split_sizes(n: int, p: int) -> List[int]:
    """numpy.array_split piece sizes: the first n mod p pieces hold one more."""
    q, rem = divmod(n, p)
    return [q + 1] * rem + [q] * (p - rem)


def adjust_groups(clusters: List[np.ndarray], M: int) -> List[np.ndarray]:
    """adjust_groups_to_target_length (Sec. 3.3): exactly M groups.

    The paper names the step but gives no rule; the reading taken:
      * C > M (merge): the cluster of rank t (ascending code) joins group
        floor(t * M / C);
      * C < M (split): D'Hondt seats with one guaranteed seat per cluster,
        each cluster cut into that many contiguous pieces in position order
        (array_split sizes);
      * C == M: unchanged."""
    C = len(clusters)
    if C == M:
        return [c.copy() for c in clusters]
    if C > M:
        groups: List[List[int]] = [[] for _ in range(M)]
        for t, c in enumerate(clusters):
            groups[(t * M) // C].extend(c.tolist())
        return [np.array(sorted(g), dtype=np.int64) for g in groups]
    seats = dhondt_seats([len(c) for c in clusters], M)
    out: List[np.ndarray] = []
    for c, p in zip(clusters, seats):
        start = 0
        for sz in array_split_sizes(len(c), p):
            out.append(c[start:start + sz].copy())
            start += sz
    return out


# ---------------------------------------------------------------------------
# Step 6: macro-tokens and positions (Sec. 3.4, Eq. macro_embed)
# ---------------------------------------------------------------------------


def group_position(members: np.ndarray, scheme: int) -> int:
    """Representative position of a group (Sec. 3.4): max (default); median
    read as the lower median; mean read as floor(mean + 1/2)."""
    p = np.sort(np.asarray(members, dtype=np.int64))
    n = p.size
    if scheme == POS_MAX:
        return int(p[-1])
    if scheme == POS_MEDIAN:
        return int(p[(n - 1) // 2])
    tot = int(p.sum())
    return (2 * tot + n) // (2 * n)


def aggregate_groups(X: np.ndarray, groups: List[np.ndarray], renorm: bool = True
                     ) -> np.ndarray:
    """Eq. macro_embed: the mean of the members, rescaled to the mean member
    norm.  A singleton is its token unchanged; a mean with norm < 1e-30 is not
    rescaled."""
    X = np.asarray(X, dtype=np.float64)
    out = np.empty((len(groups), X.shape[1]))
    for g, m in enumerate(groups):
        rows = X[m]
        if m.size == 1:
            out[g] = rows[0]
            continue
        mean = rows.mean(axis=0)
        if renorm:
            eta = np.linalg.norm(rows, axis=1).mean()
            nrm = np.linalg.norm(mean)
            if nrm >= 1e-30:
                mean = mean * (eta / nrm)
        out[g] = mean
    return out


def order_groups(groups: List[np.ndarray], scheme: int) -> List[int]:
    """Macro-tokens are sorted by representative position (Sec. 3.6); ties
    (possible for median and mean) go to the group with the smaller first
    token."""
    keys = [(group_position(g, scheme), int(np.min(g))) for g in groups]
    return sorted(range(len(groups)), key=lambda i: keys[i])


def _identity(X: np.ndarray, N: int) -> CompressResult:
    Xf = np.asarray(X, dtype=np.float64)
    return CompressResult(Xf.copy(), np.arange(N, dtype=np.int64),
                          np.arange(N, dtype=np.int64), {"identity": True})


def _assemble(X: np.ndarray, pf: int, pl: int, groups_abs: List[np.ndarray],
              cfg: CompressConfig) -> CompressResult:
    """Preserved first tokens, then the macro-tokens ordered by position, then
    the preserved last tokens; positions per pos_mode; token -> macro map."""
    N = X.shape[0]
    order = order_groups(groups_abs, cfg.pos_scheme)
    macro = aggregate_groups(X, [groups_abs[i] for i in order], cfg.renorm)
    M = pf + len(order) + pl
    Xt = np.empty((M, X.shape[1]))
    pos = np.empty(M, dtype=np.int64)
    t2m = np.full(N, -1, dtype=np.int64)
    for i in range(pf):
        Xt[i] = X[i]
        pos[i] = i
        t2m[i] = i
    for k, gi in enumerate(order):
        g = groups_abs[gi]
        Xt[pf + k] = macro[k]
        pos[pf + k] = group_position(g, cfg.pos_scheme)
        t2m[g] = pf + k
    for i in range(pl):
        tok = N - pl + i
        Xt[pf + len(order) + i] = X[tok]
        pos[pf + len(order) + i] = tok
        t2m[tok] = pf + len(order) + i
    if cfg.pos_mode == MODE_COMPACT:
        pos = np.arange(M, dtype=np.int64)
    return CompressResult(Xt, pos, t2m, {"identity": False})


def _region(N: int, cfg: CompressConfig) -> Tuple[int, int, int]:
    pf = max(0, min(cfg.preserve_first, N))
    pl = max(0, min(cfg.preserve_last, N - pf))
    return pf, pl, N - pf - pl


# ---------------------------------------------------------------------------
# Global backend (Algorithm 1 over the compressible region, Sec. 3.5)
# ---------------------------------------------------------------------------


def spectral_groups(Xc: np.ndarray, W: np.ndarray, b: np.ndarray, R: np.ndarray,
                    q1: np.ndarray, r: int, bits: int, M: int, tol: float = 1e-10,
                    phi32: bool = True, normalize: bool = False):
    """Algorithm 1 on one token set: features, Lanczos, Ritz vectors, SimHash,
    clusters and the exact-length adjustment.  Group members are indices into
    Xc.  Phi is rounded to float32 before Lanczos when phi32 (the precision
    the feature matrix is stored in); with normalize, Lanczos runs on the
    row-normalised operator (normalized_features), rounded likewise."""
    Phi = rff_features(Xc, W, b)
    if phi32:
        Phi = Phi.astype(np.float32).astype(np.float64)
    if normalize:
        Phi = normalized_features(Phi)[1]
        if phi32:
            Phi = Phi.astype(np.float32).astype(np.float64)
    alpha, beta, Q, r_eff = lanczos(Phi, q1[:Xc.shape[0]], r, tol)
    theta, S, U = ritz_pairs(alpha, beta, Q)
    codes = simhash(U.astype(np.float32), R[:bits, :r_eff])
    clusters = bucket(codes)
    groups = adjust_groups(clusters, M)
    info = {"theta": theta, "alpha": alpha, "beta": beta, "r_eff": r_eff,
            "codes": codes, "n_clusters": len(clusters), "U": U, "Q": Q}
    return groups, info


def compress_global(X: np.ndarray, W: np.ndarray, b: np.ndarray, R: np.ndarray,
                    q1: np.ndarray, cfg: CompressConfig) -> CompressResult:
    """The global-LSH backend (Sec. 3.5): Spectral-LSH over the compressible
    region [pf, N - pl), preserved tokens kept as singletons; rho <= 1 or an
    empty region is the exact identity (Sec. 5.6, App. B.6)."""
    X = np.asarray(X, dtype=np.float64)
    N = X.shape[0]
    pf, pl, Nc = _region(N, cfg)
    if cfg.rho <= 1.0 or Nc <= 0:
        return _identity(X, N)
    M = target_count(Nc, cfg.rho)
    bits = cfg.bits if cfg.bits > 0 else auto_bits(Nc, cfg.rho)
    groups, info = spectral_groups(X[pf:N - pl], W, b, R, q1, cfg.r, bits, M,
                                   cfg.lanczos_tol, normalize=cfg.normalize)
    res = _assemble(X, pf, pl, [g + pf for g in groups], cfg)
    res.info.update(info)
    res.info.update({"M_star": M, "bits": bits})
    return res


def compress_chunk(X: np.ndarray, cfg: CompressConfig) -> CompressResult:
    """Chunk backend (Sec. 3.5): consecutive groups of k = max(1, round(rho))
    tokens over the compressible region, aggregated like any group."""
    X = np.asarray(X, dtype=np.float64)
    N = X.shape[0]
    pf, pl, Nc = _region(N, cfg)
    if cfg.rho <= 1.0 or Nc <= 0:
        return _identity(X, N)
    k = max(1, int(round(cfg.rho)))
    groups = [np.arange(s, min(s + k, Nc)) + pf for s in range(0, Nc, k)]
    return _assemble(X, pf, pl, groups, cfg)


# ---------------------------------------------------------------------------
# Adaptive backend (Sec. 3.6, App. B.8)
# ---------------------------------------------------------------------------


def tau_schedule(rho: float) -> float:
    """Threshold tau(rho): 0.70 at rho=2, 0.60 at rho=8, 0.55 at rho=16
    (Sec. 3.6).  The paper says the schedule interpolates; all three points lie
    on 0.75 - 0.05 log2(rho), clamped to [0.55, 0.70], which is the reading."""
    t = 0.75 - 0.05 * math.log2(rho)
    return min(0.70, max(0.55, t))


def redundancy_score(Xw: np.ndarray) -> float:
    """Eq. redundancy: the mean cosine between each token and the
    L2-normalised centroid of the window.  A zero-norm token contributes 0; a
    zero centroid gives 0."""
    Xw = np.asarray(Xw, dtype=np.float64)
    L = Xw.shape[0]
    c = Xw.mean(axis=0)
    cn = np.linalg.norm(c)
    if cn == 0.0:
        return 0.0
    c = c / cn
    tot = 0.0
    for i in range(L):
        n = np.linalg.norm(Xw[i])
        if n > 0.0:
            tot += float(Xw[i] @ c) / n
    return tot / L


def window_bounds(Nc: int, w: int) -> List[Tuple[int, int]]:
    """Consecutive windows of w tokens over the region; the last is shorter."""
    return [(s, min(s + w, Nc)) for s in range(0, Nc, w)]


def window_budgets(lengths: Sequence[int], M: int) -> List[int]:
    """Exact per-window output budgets summing to M (Sec. 3.6, App. B.8).

    The paper gives no rule; the reading: every window first receives one
    macro-token, and the remaining E = M - W are apportioned by largest
    remainder (Hamilton) over quotas E (L_w - 1) / (N_c - W), remainders
    compared exactly as integers, ties to the lower window index.  This keeps
    1 <= m_w <= L_w.  Requires W <= M <= N_c."""
    W = len(lengths)
    Nc = int(sum(lengths))
    assert W <= M <= Nc
    E = M - W
    den = Nc - W
    if den == 0 or E == 0:
        return [1] * W
    base = [(E * (L - 1)) // den for L in lengths]
    rem = [(E * (L - 1)) % den for L in lengths]
    left = E - sum(base)
    order = sorted(range(W), key=lambda i: (-rem[i], i))
    out = [1 + x for x in base]
    for i in order[:left]:
        out[i] += 1
    return out


def route_windows(X: np.ndarray, bounds: List[Tuple[int, int]], rho: float,
                  cfg: CompressConfig) -> Tuple[List[bool], List[float]]:
    """Routing policy (Sec. 3.6): at rho >= 16 every window is spectral
    (routing bypassed); otherwise L <= 4 -> chunk, score < tau -> chunk, else
    spectral.  Returns (spectral flags, scores)."""
    tau = tau_schedule(rho) if cfg.tau_schedule else cfg.tau
    spectral, scores = [], []
    for (s, e) in bounds:
        L = e - s
        sc = redundancy_score(X[s:e])
        scores.append(sc)
        if rho >= 16.0:
            spectral.append(True)
        elif L <= 4:
            spectral.append(False)
        else:
            spectral.append(sc >= tau)
    return spectral, scores


def chunk_groups(L: int, m: int) -> List[np.ndarray]:
    """The chunk compressor with an exact budget: m contiguous groups with
    array_split sizes."""
    out, start = [], 0
    for sz in array_split_sizes(L, m):
        out.append(np.arange(start, start + sz))
        start += sz
    return out


def _windowed(X: np.ndarray, W: np.ndarray, b: np.ndarray, R: np.ndarray,
              q1: np.ndarray, cfg: CompressConfig, route: bool) -> CompressResult:
    """Consecutive windows of cfg.window tokens over the compressible region,
    exact per-window budgets (App. B.8), each window either chunk-averaged or
    compressed by Spectral-LSH on its own tokens, macro-tokens concatenated in
    window order.  route=False sends every window down the spectral path."""
    X = np.asarray(X, dtype=np.float64)
    N = X.shape[0]
    pf, pl, Nc = _region(N, cfg)
    if cfg.rho <= 1.0 or Nc <= 0:
        return _identity(X, N)
    M = target_count(Nc, cfg.rho)
    Xc = X[pf:N - pl]
    bounds = window_bounds(Nc, cfg.window)
    budgets = window_budgets([e - s for s, e in bounds], M)
    if route:
        spectral, scores = route_windows(Xc, bounds, cfg.rho, cfg)
    else:
        spectral, scores = [True] * len(bounds), []
    groups_abs: List[np.ndarray] = []
    r_effs = []
    for (s, e), m, sp in zip(bounds, budgets, spectral):
        L = e - s
        if sp:
            bits = cfg.bits if cfg.bits > 0 else auto_bits(L, cfg.rho)
            gs, inf = spectral_groups(Xc[s:e], W, b, R, q1[s:e], cfg.r, bits, m,
                                      cfg.lanczos_tol, normalize=cfg.normalize)
            r_effs.append(inf["r_eff"])
        else:
            gs = chunk_groups(L, m)
            r_effs.append(0)
        groups_abs.extend(g + s + pf for g in gs)
    res = _assemble(X, pf, pl, groups_abs, cfg)
    res.info.update({"M_star": M, "budgets": budgets, "spectral": spectral,
                     "scores": scores, "r_eff": r_effs})
    return res


def compress_adaptive(X: np.ndarray, W: np.ndarray, b: np.ndarray, R: np.ndarray,
                      q1: np.ndarray, cfg: CompressConfig) -> CompressResult:
    """Adaptive backend (Sec. 3.6): windows, exact budgets, redundancy score,
    chunk or per-window Spectral-LSH, concatenation in window order.  Each
    spectral window uses the slice of q1 at its offset and
    b_w = cfg.bits or ceil(log2(L_w / rho))."""
    return _windowed(X, W, b, R, q1, cfg, route=True)


def compress_local(X: np.ndarray, W: np.ndarray, b: np.ndarray, R: np.ndarray,
                   q1: np.ndarray, cfg: CompressConfig) -> CompressResult:
    """Local-LSH backend (Sec. 3.5): Spectral-LSH run independently inside
    each window of cfg.window tokens (the paper's default window is 16), with
    the exact per-window budgets of the adaptive backend and no routing; the
    adaptive backend at rho >= 16 delegates to exactly this (Sec. 3.6)."""
    return _windowed(X, W, b, R, q1, cfg, route=False)


# ---------------------------------------------------------------------------
# Cost model (Sec. 3.7)
# ---------------------------------------------------------------------------


def complexity_ops(d: int, D: int, r: int, b: int) -> int:
    """Operations per token of the spectral path, D (d + r) + r b (Sec. 3.7)."""
    return D * (d + r) + r * b

"""Helpers shared by the GPU parity tests: seeded inputs as torch tensors and
the comparison metrics.  Inputs come from the workload generator; expected
values come only from the CPU oracle."""
import math

import numpy as np
import scipy.linalg
import torch

import oracle as O
import workloads as WL


def to_torch_x(prompt_or_bits, dtype, device="cuda"):
    """Embeddings / W from the generator: float32 arrays or bf16 bit patterns."""
    a = prompt_or_bits
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(device)


def widen(a, dtype):
    return WL.bf16_bits_to_f32(a).astype(np.float64) if dtype == "bf16" else a.astype(np.float64)


def feature_tolerance(X64, W64, b64):
    """Per-element bound for a float32 evaluation of Eq. rff_map: the
    contraction in float32 (error within a small multiple of 2^-24 times
    sum_k |x_k w_k|), the rounded sum with b and the float32 cosine and scale
    (a few units of 2^-24 of 1 + |theta|); 2^-20 leaves a factor of 16."""
    D = W64.shape[0]
    theta = X64 @ W64.T + b64[None, :]
    S = np.abs(X64) @ np.abs(W64).T
    return math.sqrt(2.0 / D) * 2.0 ** -20 * (4.0 + np.abs(theta) + S)


def max_subspace_angle(A, B):
    return float(np.max(scipy.linalg.subspace_angles(np.asarray(A, np.float64),
                                                     np.asarray(B, np.float64))))


def oracle_phi32(X64, W64, b):
    return O.rff_features(X64, W64, b).astype(np.float32)


def pinned(t):
    return t.pin_memory() if torch.cuda.is_available() else t


def adjusted_rand_index(a, b):
    """Adjusted Rand index of two labelings of the same items (Hubert and
    Arabie, 1985): the pair-counting agreement of the two partitions,
    corrected for chance; 1 for identical partitions."""
    a = np.asarray(a, np.int64)
    b = np.asarray(b, np.int64)
    n = a.size
    _, ia = np.unique(a, return_inverse=True)
    _, ib = np.unique(b, return_inverse=True)
    pair = ia * (int(ib.max()) + 1) + ib
    _, nij = np.unique(pair, return_counts=True)
    comb = lambda x: x.astype(np.float64) * (x - 1) / 2.0
    s_ij = comb(nij).sum()
    s_a = comb(np.bincount(ia)).sum()
    s_b = comb(np.bincount(ib)).sum()
    tot = n * (n - 1) / 2.0
    expected = s_a * s_b / tot if tot > 0 else 0.0
    top = 0.5 * (s_a + s_b)
    if top == expected:
        return 1.0
    return float((s_ij - expected) / (top - expected))


def code_agreement(sls, w, p, prm, X, Wt, bt, Rt, qt):
    """End-to-end agreement of the GPU pass with the oracle's
    compress_global on one prompt (reported, not pinned: float32 against
    float64 Ritz vectors flip near-zero SimHash dots): the fraction of
    identical codes (GPU codes from the same feature, Lanczos and SimHash
    kernels sls_compress runs) and the adjusted Rand index of the two token
    maps.  Returns a dict."""
    Nc = w.N - w.preserve_first - w.preserve_last
    cfg_o = O.CompressConfig(rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                             preserve_first=w.preserve_first, preserve_last=w.preserve_last)
    res = O.compress_global(p.x_f64(), prm.w_f64(), prm.b, prm.R, prm.q1, cfg_o)
    codes_o = res.info["codes"]
    bits = res.info["bits"]
    Xc = X[w.preserve_first:w.preserve_first + Nc]
    phi = sls.feature_map(Xc, Wt, bt)
    _, U, r_eff, _, _ = sls.lanczos_topr(phi, qt[:Nc], w.r)
    codes_g = sls.simhash(U, Rt, bits, k_dev=r_eff).cpu().numpy().view(np.uint32)
    cfg = sls.Config.make(backend=sls.BACKEND_GLOBAL, rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                          preserve_first=w.preserve_first, preserve_last=w.preserve_last)
    _, _, t2m, _, _ = sls.compress(X.view(1, w.N, w.d), cfg, Wt, bt, Rt, qt)
    t2m = t2m[0].cpu().numpy()
    return {"workload": w.name, "tokens": Nc,
            "codes_identical": float(np.mean(codes_g == codes_o)),
            "ari_tok2macro": adjusted_rand_index(t2m, res.tok2macro),
            "clusters_gpu": int(np.unique(codes_g).size),
            "clusters_oracle": int(res.info["n_clusters"])}

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

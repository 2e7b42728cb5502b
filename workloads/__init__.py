"""Seeded synthetic inputs for the Spectral-LSH compression pass.

This module is shared by the tests, the benchmark and the CPU oracle's checks.
It holds no arithmetic of the method itself: it only draws token ids, looks up
rows of a Gaussian "vocabulary" table, and draws the random parameters the
method consumes (Omega, b, the SimHash hyperplanes R and the Lanczos start
vector q1).  Both the CUDA path and the oracle receive exactly these arrays, so
they see identical randomness.

Workload recipes (prompt embeddings stand in for the C4 / Wikitext prompts and
the LLM embedding tables of the paper's experiments, Sec. 5.1, which are not
available here):

* ``tiny``      N=512,  d=64,   V=2000,   Zipf(1.1), fp32, plus N(0, 0.01) noise
* ``mistral7b`` N=8192, d=4096, V=32768,  Zipf(1.1), bf16, 64-token spans
                copied from earlier positions until ~20% of tokens are copies
* ``qwen7b``    N=32768, d=3584, V=151936, Zipf(1.05), bf16, spans of length
                U[16, 256] copied until ~30% are copies
* ``qwen14b``   N=131072, d=5120, V=151936, Zipf(1.05), bf16, periodic templates
                (period U[8, 64]) over ~40% of the sequence (the JSON/code/
                table-like structure of the paper's stress test, Table 4)
* ``adaptive``  64 prompts of N=16384, d=4096, bf16, generated like
                ``mistral7b`` with duplication 0.6*p/63 for prompt p.
* ``local``     the ``qwen7b`` prompt at the paper's local-LSH defaults
                (Sec. 5.1 hyperparameters: D=256, r=16, window 16, bits from
                the window budget), rho=8.
* ``adaptive_mixed`` 64 prompts of N=16384, d=4096, bf16 (the ``adaptive``
                vocabulary, no copied spans) in which each 2048-token window
                of the compressible region is, with probability 1/2 (seeded),
                a coherent window: its rows are 0.8 t + 0.6 e_i with t a unit
                topic direction drawn for the window and e_i the token's
                vocabulary row.  A coherent window's tokens share a direction
                (redundancy score about 0.8 on Eq. redundancy) while keeping
                full rank; the others score near 0, so the adaptive router
                sends about half of the windows to the spectral chain and half
                to the chunk path at rho = 4 and 8.

Vocabulary rows are N(0, 1/d) and are produced by a counter-based generator
(numpy Philox keyed by the seed, counter = token id), so the V x d table is
never materialised and a row depends only on (seed, id).

All draws use numpy's Philox bit generator; data seed 0, parameter seed 1.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

DATA_SEED = 0
PARAM_SEED = 1

# ---------------------------------------------------------------------------
# bf16 helpers (storage format only; round-to-nearest-even from float32)
# ---------------------------------------------------------------------------


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); return the
    16-bit patterns as uint16.  NaNs are kept quiet NaNs."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    rounding_bias = ((u >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    r = ((u + rounding_bias) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        r[nan] = 0x7FC0
    return r


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns (uint16) to float32 exactly."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------------------
# Random sources
# ---------------------------------------------------------------------------


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(key=[seed, stream]))


_STREAM_IDS = 11
_STREAM_SPANS = 12
_STREAM_NOISE = 13
_STREAM_TOPIC = 14
_STREAM_W = 21
_STREAM_B = 22
_STREAM_R = 23
_STREAM_Q = 24
_VOCAB_KEY = 0x766F636162  # "vocab"


def vocab_rows(seed: int, ids: np.ndarray, d: int) -> np.ndarray:
    """Rows of the seeded Gaussian table, N(0, 1/d) entries, float64.

    Row ``v`` is drawn from Philox(key=(seed, VOCAB_KEY), counter=(0, v, 0, 0)),
    so it depends only on (seed, v)."""
    ids = np.asarray(ids, dtype=np.int64)
    uniq, inv = np.unique(ids, return_inverse=True)
    table = np.empty((uniq.size, d), dtype=np.float64)
    scale = 1.0 / math.sqrt(d)
    for k, v in enumerate(uniq):
        g = np.random.Generator(
            np.random.Philox(key=[seed, _VOCAB_KEY], counter=[0, int(v), 0, 0]))
        table[k] = g.standard_normal(d) * scale
    return table[inv]


def zipf_ids(rng: np.random.Generator, n: int, V: int, s: float) -> np.ndarray:
    """Token ids with p(k) proportional to k^-s over k = 1..V (finite support),
    returned as k - 1."""
    k = np.arange(1, V + 1, dtype=np.float64)
    p = k ** (-s)
    cdf = np.cumsum(p)
    cdf /= cdf[-1]
    u = rng.random(n)
    return np.minimum(np.searchsorted(cdf, u, side="right"), V - 1).astype(np.int64)


def copy_spans(rng: np.random.Generator, ids: np.ndarray, frac: float,
               span_lo: int, span_hi: int) -> np.ndarray:
    """Overwrite spans with copies of earlier spans until ``frac`` of the
    tokens are copies (exact duplicates of an earlier token sequence)."""
    ids = ids.copy()
    n = ids.size
    if frac <= 0 or n < 2 * span_lo:
        return ids
    copied = np.zeros(n, dtype=bool)
    target = frac * n
    guard = 0
    while copied.sum() < target and guard < 100000:
        guard += 1
        L = int(rng.integers(span_lo, span_hi + 1))
        L = min(L, n // 2)
        dst = int(rng.integers(L, n - L + 1))
        src = int(rng.integers(0, dst - L + 1))
        ids[dst:dst + L] = ids[src:src + L]
        copied[dst:dst + L] = True
    return ids


def periodic_templates(rng: np.random.Generator, ids: np.ndarray, frac: float,
                       V: int, s: float, per_lo: int = 8, per_hi: int = 64,
                       reg_lo: int = 256, reg_hi: int = 4096) -> np.ndarray:
    """Overwrite regions with a short Zipf-drawn id pattern repeated with period
    U[per_lo, per_hi] until ``frac`` of the tokens lie in such regions."""
    ids = ids.copy()
    n = ids.size
    covered = np.zeros(n, dtype=bool)
    target = frac * n
    guard = 0
    while covered.sum() < target and guard < 100000:
        guard += 1
        P = int(rng.integers(per_lo, per_hi + 1))
        L = int(rng.integers(reg_lo, reg_hi + 1))
        L = min(L, n)
        start = int(rng.integers(0, n - L + 1))
        pattern = zipf_ids(rng, P, V, s)
        ids[start:start + L] = np.resize(pattern, L)
        covered[start:start + L] = True
    return ids


# ---------------------------------------------------------------------------
# Workload descriptions
# ---------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    N: int              # tokens per prompt
    d: int              # embedding width
    V: int              # vocabulary size
    zipf: float
    dtype: str          # "f32" or "bf16"
    D: int              # RFF features
    r: int              # Krylov rank
    bits: int           # SimHash bits (0 = ceil(log2(N_c / rho)))
    rho: float          # target compression
    preserve_first: int = 0
    preserve_last: int = 12
    noise_var: float = 0.0
    dup_frac: float = 0.0
    span_lo: int = 64
    span_hi: int = 64
    template_frac: float = 0.0
    batch: int = 1      # independent prompts (adaptive workload)
    window: int = 0     # window length of the windowed backends (0 = global backend)
    rhos: tuple = ()    # swept compression ratios (adaptive workload)
    backend: str = "global"   # "global", "adaptive" or "local"
    coherent_frac: float = 0.0  # share of coherent windows (adaptive_mixed)
    coherent_mix: float = 0.8   # weight of the window's topic direction in them


WORKLOADS = {
    "tiny": Workload("tiny", N=512, d=64, V=2000, zipf=1.1, dtype="f32",
                     D=256, r=16, bits=8, rho=4.0, noise_var=0.01),
    "mistral7b": Workload("mistral7b", N=8192, d=4096, V=32768, zipf=1.1,
                          dtype="bf16", D=1024, r=32, bits=12, rho=8.0,
                          dup_frac=0.2, span_lo=64, span_hi=64),
    "qwen7b": Workload("qwen7b", N=32768, d=3584, V=151936, zipf=1.05,
                       dtype="bf16", D=2048, r=64, bits=16, rho=16.0,
                       dup_frac=0.3, span_lo=16, span_hi=256),
    "qwen14b": Workload("qwen14b", N=131072, d=5120, V=151936, zipf=1.05,
                        dtype="bf16", D=2048, r=64, bits=16, rho=16.0,
                        template_frac=0.4),
    "adaptive": Workload("adaptive", N=16384, d=4096, V=32768, zipf=1.1,
                         dtype="bf16", D=1024, r=32, bits=0, rho=8.0,
                         dup_frac=0.0, span_lo=64, span_hi=64, batch=64,
                         window=2048, rhos=(2.0, 4.0, 8.0, 16.0), backend="adaptive"),
    "adaptive_mixed": Workload("adaptive_mixed", N=16384, d=4096, V=32768, zipf=1.1,
                               dtype="bf16", D=1024, r=32, bits=0, rho=8.0,
                               dup_frac=0.0, span_lo=64, span_hi=64, batch=64,
                               window=2048, rhos=(4.0, 8.0), backend="adaptive",
                               coherent_frac=0.5),
    "local": Workload("local", N=32768, d=3584, V=151936, zipf=1.05,
                      dtype="bf16", D=256, r=16, bits=0, rho=8.0,
                      dup_frac=0.3, span_lo=16, span_hi=256, window=16,
                      backend="local"),
}


def scaled(w: Workload, **kw) -> Workload:
    """A copy of a workload with some fields replaced (smaller parity cases)."""
    return dataclasses.replace(w, **kw)


@dataclasses.dataclass
class Prompt:
    ids: np.ndarray          # (N,) int64
    X: np.ndarray            # (N, d) float32, or uint16 bf16 bit patterns
    dtype: str               # "f32" | "bf16"

    def x_f64(self) -> np.ndarray:
        """Exact float64 widening of the stored embeddings."""
        if self.dtype == "bf16":
            return bf16_bits_to_f32(self.X).astype(np.float64)
        return self.X.astype(np.float64)


def prompt_ids(w: Workload, seed: int = DATA_SEED, index: int = 0,
               dup_frac: Optional[float] = None) -> np.ndarray:
    rng = _rng(seed + 1000 * index, _STREAM_IDS)
    ids = zipf_ids(rng, w.N, w.V, w.zipf)
    srng = _rng(seed + 1000 * index, _STREAM_SPANS)
    frac = w.dup_frac if dup_frac is None else dup_frac
    if frac > 0:
        ids = copy_spans(srng, ids, frac, w.span_lo, w.span_hi)
    if w.template_frac > 0:
        ids = periodic_templates(srng, ids, w.template_frac, w.V, w.zipf)
    return ids


def coherent_windows(w: Workload, seed: int = DATA_SEED, index: int = 0):
    """The coherent windows of prompt ``index`` of a workload with
    coherent_frac > 0: a list of (row start, row end, unit topic direction t)
    over the windows of the compressible region [preserve_first, N -
    preserve_last), each window coherent with probability coherent_frac."""
    if w.coherent_frac <= 0 or w.window <= 0:
        return []
    rng = _rng(seed + 1000 * index, _STREAM_TOPIC)
    pf, nc = w.preserve_first, w.N - w.preserve_first - w.preserve_last
    out = []
    for s0 in range(0, nc, w.window):
        pick = rng.random() < w.coherent_frac
        t = rng.standard_normal(w.d)
        if pick:
            out.append((pf + s0, pf + min(s0 + w.window, nc), t / np.linalg.norm(t)))
    return out


def make_prompt(w: Workload, seed: int = DATA_SEED, index: int = 0,
                dup_frac: Optional[float] = None) -> Prompt:
    ids = prompt_ids(w, seed, index, dup_frac)
    if w.coherent_frac > 0:
        X = vocab_rows(seed, ids, w.d)
        a = w.coherent_mix
        for r0, r1, t in coherent_windows(w, seed, index):
            X[r0:r1] = a * t[None, :] + math.sqrt(1.0 - a * a) * X[r0:r1]
        X32 = X.astype(np.float32)
        return Prompt(ids, f32_to_bf16_bits(X32) if w.dtype == "bf16" else X32, w.dtype)
    uniq, inv = np.unique(ids, return_inverse=True)
    table = vocab_rows(seed, uniq, w.d).astype(np.float32)
    if w.noise_var > 0:
        X = table[inv].astype(np.float64)
        nrng = _rng(seed + 1000 * index, _STREAM_NOISE)
        X += nrng.standard_normal(X.shape) * math.sqrt(w.noise_var)
        X32 = X.astype(np.float32)
        if w.dtype == "bf16":
            return Prompt(ids, f32_to_bf16_bits(X32), "bf16")
        return Prompt(ids, X32, "f32")
    if w.dtype == "bf16":
        return Prompt(ids, f32_to_bf16_bits(table)[inv], "bf16")
    return Prompt(ids, table[inv], "f32")


def adaptive_dup_frac(p: int, batch: int) -> float:
    """Duplication fraction of prompt p in the adaptive batch: 0.6 * p / (B-1)."""
    return 0.0 if batch <= 1 else 0.6 * p / (batch - 1)


@dataclasses.dataclass
class Params:
    """Random draws consumed by the method (Sec. 3.2 and Sec. 3.3)."""
    W: np.ndarray    # (D, d) = Omega^T; float32 or bf16 bits (same as X)
    b: np.ndarray    # (D,) float32, U(0, 2 pi)
    R: np.ndarray    # (bits_max, r) float32, N(0, 1)
    q1: np.ndarray   # (n_q,) float64, N(0, 1)
    dtype: str

    def w_f64(self) -> np.ndarray:
        if self.dtype == "bf16":
            return bf16_bits_to_f32(self.W).astype(np.float64)
        return self.W.astype(np.float64)


def make_params(D: int, d: int, r: int, bits_max: int, n_q: int, dtype: str,
                seed: int = PARAM_SEED) -> Params:
    """W ~ N(0, 1/sqrt(d)) (variance), rounded to the embedding dtype;
    b ~ U(0, 2 pi); R ~ N(0, 1); q1 ~ N(0, 1)."""
    gw = _rng(seed, _STREAM_W)
    W = gw.standard_normal((D, d)) * (d ** -0.25)
    W32 = W.astype(np.float32)
    Wst = f32_to_bf16_bits(W32) if dtype == "bf16" else W32
    gb = _rng(seed, _STREAM_B)
    b = (gb.random(D) * (2.0 * math.pi)).astype(np.float32)
    gr = _rng(seed, _STREAM_R)
    R = gr.standard_normal((max(1, bits_max), r)).astype(np.float32)
    gq = _rng(seed, _STREAM_Q)
    q1 = gq.standard_normal(max(1, n_q))
    return Params(Wst, b, R, q1, dtype)


def params_for(w: Workload, seed: int = PARAM_SEED) -> Params:
    n_q = w.N if w.batch == 1 else w.batch * w.N
    return make_params(w.D, w.d, w.r, 32, n_q, w.dtype, seed)

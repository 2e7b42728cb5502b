"""GB300 (sm_103a) Spectral-LSH compression pass (arXiv 2607.19368).

Thin Python binding of the C ABI in ``include/sls.h`` (``libsls.so``).  Every
step of the pass runs in the library's CUDA kernels; this module only
marshals torch tensors (device memory and the current stream) into the C
calls and raises on a non-zero status.  There is no CPU fallback: if the
library is not built, importing the functions works but every call raises.

The same names as the C entry points are exported:
``feature_map``, ``lanczos_topr``, ``simhash``, ``aggregate``, ``compress``,
``embed_gather``, ``compress_tokens``.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

__all__ = [
    "SLS_OK", "SLS_F32", "SLS_BF16", "POS_MAX", "POS_MEDIAN", "POS_MEAN",
    "MODE_REPRESENTATIVE", "MODE_COMPACT", "BACKEND_GLOBAL", "BACKEND_ADAPTIVE",
    "BACKEND_CHUNK", "BACKEND_LOCAL", "Config", "SLSError", "lib", "lib_path", "feature_map",
    "feature_map_batched", "feature_normalize",
    "lanczos_topr", "simhash", "aggregate", "compress", "output_count",
    "compress_workspace_size", "workspace_status", "EXPORTED", "PHASES",
    "set_phase_events", "launch_count", "Workspace", "embed_gather", "compress_tokens",
    "compress_tokens_workspace_size", "TokensWorkspace", "selftest_wait_limit",
    "lanczos_topr_batched", "selftest_lanczos_giveup",
]

SLS_OK = 0
SLS_F32, SLS_BF16 = 0, 1
POS_MAX, POS_MEDIAN, POS_MEAN = 0, 1, 2
MODE_REPRESENTATIVE, MODE_COMPACT = 0, 1
BACKEND_GLOBAL, BACKEND_ADAPTIVE, BACKEND_CHUNK, BACKEND_LOCAL = 0, 1, 2, 3

_HERE = os.path.dirname(os.path.abspath(__file__))


def lib_path() -> str:
    """The library the binding loads: libsls.so next to this file, or the
    path in the SLS_LIBRARY environment variable (e.g. the debug build
    libsls_debug.so), read when the library is first loaded."""
    return os.environ.get("SLS_LIBRARY") or os.path.join(_HERE, "libsls.so")


def debug_lib_path() -> str:
    return os.path.join(_HERE, "libsls_debug.so")


# With SLS_CHECK_STATUS=1 every call that takes a workspace reads its status
# word afterwards (synchronising) and raises on anything but SLS_OK: with the
# debug build this turns each call into a bounds and guard-band check.
_CHECK_STATUS = os.environ.get("SLS_CHECK_STATUS") == "1"


def _check_ws(fn: str, ws: torch.Tensor):
    if _CHECK_STATUS:
        st = int(lib().sls_workspace_status(_ptr(ws), _stream(ws)))
        if st != SLS_OK:
            raise SLSError(fn + " (device status)", st, lib().sls_status_string(st).decode())


class SLSError(RuntimeError):
    """A libsls call returned a non-zero status."""

    def __init__(self, fn: str, status: int, text: str):
        super().__init__(f"{fn}: status {status} ({text})")
        self.status = status


class Config(ctypes.Structure):
    """sls_config_t: the fields of the paper's CompressionConfig (App. B.3)."""
    _fields_ = [
        ("backend", ctypes.c_int), ("rho", ctypes.c_double), ("D", ctypes.c_int),
        ("r", ctypes.c_int), ("bits", ctypes.c_int), ("preserve_first", ctypes.c_int),
        ("preserve_last", ctypes.c_int), ("pos_scheme", ctypes.c_int),
        ("pos_mode", ctypes.c_int), ("renorm", ctypes.c_int),
        ("lanczos_tol", ctypes.c_double), ("window", ctypes.c_int),
        ("tau", ctypes.c_double), ("tau_schedule", ctypes.c_int),
        ("normalize", ctypes.c_int), ("phi_dtype", ctypes.c_int),
    ]

    @classmethod
    def make(cls, backend=BACKEND_GLOBAL, rho=4.0, D=256, r=16, bits=0, preserve_first=0,
             preserve_last=12, pos_scheme=POS_MAX, pos_mode=MODE_REPRESENTATIVE, renorm=1,
             lanczos_tol=1e-10, window=2048, tau=0.70, tau_schedule=1,
             normalize=0, phi_dtype=SLS_F32) -> "Config":
        """phi_dtype: storage of the feature matrix, SLS_F32 or SLS_BF16."""
        return cls(backend, float(rho), D, r, bits, preserve_first, preserve_last, pos_scheme,
                   pos_mode, int(renorm), float(lanczos_tol), window, float(tau),
                   int(tau_schedule), int(normalize), int(phi_dtype))


class _Params(ctypes.Structure):
    _fields_ = [
        ("W", ctypes.c_void_p), ("b", ctypes.c_void_p), ("R", ctypes.c_void_p),
        ("R_rows", ctypes.c_int), ("R_ld", ctypes.c_int), ("q1", ctypes.c_void_p),
        ("q1_stride", ctypes.c_int64),
    ]


_vp, _i64, _i32, _sz, _d = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_size_t,
                            ctypes.c_double)

# name -> (restype, argtypes); the exported surface of include/sls.h
EXPORTED = {
    "sls_status_string": (ctypes.c_char_p, [_i32]),
    "sls_version": (_i32, []),
    "sls_feature_map": (_i32, [_vp, _i32, _i64, _i32, _i64, _vp, _vp, _i32, _vp, _vp]),
    "sls_feature_map_ex": (_i32, [_vp, _i32, _i64, _i32, _i64, _vp, _vp, _i32, _vp, _i32, _vp]),
    "sls_lanczos_topr_ex": (_i32, [_vp, _i32, _i64, _i32, _i32, _vp, _d, _vp, _vp, _vp, _vp,
                                   _vp, _vp, _sz, _vp]),
    "sls_feature_normalize_workspace_size": (ctypes.c_size_t, [_i64, _i32]),
    "sls_feature_normalize": (_i32, [_vp, _i64, _i32, _vp, _vp, ctypes.c_size_t, _vp]),
    "sls_feature_map_batched": (_i32, [_vp, _i64, _i64, _i64, _i32, _i64, _vp, _vp, _i32, _vp,
                                       _vp, _i32, _i32, _vp]),
    "sls_lanczos_workspace_size": (_sz, [_i64, _i32, _i32]),
    "sls_lanczos_topr": (_i32, [_vp, _i64, _i32, _i32, _vp, _d, _vp, _vp, _vp, _vp, _vp, _vp,
                                _sz, _vp]),
    "sls_simhash": (_i32, [_vp, _i64, _i32, _i32, _vp, _vp, _i32, _i32, _vp, _vp]),
    "sls_aggregate_workspace_size": (_sz, [_i64, _i32, _i64]),
    "sls_aggregate": (_i32, [_vp, _i32, _i64, _i32, _i64, _vp, _i64, _i32, _i32, _vp, _vp, _vp,
                             _vp, _sz, _vp]),
    "sls_output_count": (_i64, [ctypes.POINTER(Config), _i64]),
    "sls_compress_workspace_size": (_sz, [ctypes.POINTER(Config), _i64, _i64, _i32]),
    "sls_compress": (_i32, [ctypes.POINTER(Config), _vp, _i32, _i64, _i64, _i32, _i64,
                            ctypes.POINTER(_Params), _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "sls_workspace_status": (_i32, [_vp, _vp]),
    "sls_selftest_wait_limit": (_i32, [_i32, _vp, _sz, _vp]),
    "sls_embed_gather": (_i32, [_vp, _i32, _i64, _i32, _i64, _vp, _i64, _vp, _i64, _vp, _vp]),
    "sls_compress_tokens_workspace_size": (_sz, [ctypes.POINTER(Config), _i32, _i64, _i64,
                                                 _i32]),
    "sls_compress_tokens": (_i32, [ctypes.POINTER(Config), _vp, _i32, _i64, _i32, _i64, _vp,
                                   _i64, _i64, ctypes.POINTER(_Params), _vp, _vp, _vp, _vp, _vp,
                                   _vp, _vp, _sz, _vp]),
    "sls_lanczos_topr_noalloc": (_i32, [_vp, _i64, _i32, _i32, _vp, _d, _vp, _vp, _vp, _vp,
                                        _vp, _vp]),
    "sls_lanczos_batched_workspace_size": (_sz, [_i64, _i64, _i32, _i32, _i32]),
    "sls_lanczos_topr_batched": (_i32, [_vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _i64, _i64,
                                        _vp, _d, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "sls_selftest_lanczos_giveup": (_i32, [_vp, _i64, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _sz,
                                           _vp]),
    "sls_debug_selftest": (_i32, [_i32, _vp, _sz, _vp]),
    "sls_set_phase_events": (_i32, [ctypes.POINTER(ctypes.c_void_p), _i32]),
    "sls_launch_count": (_i64, []),
}

PHASES = ("setup", "features", "lanczos", "ritz", "simhash", "segment", "aggregate")

_lib = None


def lib() -> ctypes.CDLL:
    """Load libsls.so (built by ``python -m paper_2607_19368_gb300.build``)."""
    global _lib
    if _lib is None:
        path = lib_path()
        if not os.path.exists(path):
            raise RuntimeError(
                f"{path} is missing: build the CUDA library first "
                "(python -m paper_2607_19368_gb300.build); there is no CPU fallback")
        L = ctypes.CDLL(path)
        for name, (res, args) in EXPORTED.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(fn: str, st: int):
    if st != SLS_OK:
        raise SLSError(fn, st, lib().sls_status_string(st).decode())


def _stream(t: torch.Tensor):
    return ctypes.c_void_p(torch.cuda.current_stream(t.device).cuda_stream)


def _ptr(t: Optional[torch.Tensor]):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return SLS_F32
    if t.dtype == torch.bfloat16:
        return SLS_BF16
    raise TypeError(f"unsupported embedding dtype {t.dtype} (float32 or bfloat16)")


def _need_cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise ValueError("libsls works on CUDA tensors only (no CPU fallback)")


def _workspace(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def feature_map(X: torch.Tensor, W: torch.Tensor, b: torch.Tensor,
                out: Optional[torch.Tensor] = None,
                phi_dtype: torch.dtype = torch.float32) -> torch.Tensor:
    """Phi = sqrt(2/D) cos(X W^T + b) (Sec. 3.2, Eq. rff_map); X is N x d,
    W = Omega^T is D x d (same dtype), b has D floats.  Returns N x D in
    phi_dtype: float32, or bfloat16 (each feature rounded to nearest even)."""
    _need_cuda(X, W, b)
    N, d = X.shape
    D = W.shape[0]
    assert W.shape[1] == d and W.dtype == X.dtype and W.is_contiguous()
    if out is None:
        out = torch.empty((N, D), dtype=phi_dtype, device=X.device)
    st = lib().sls_feature_map_ex(_ptr(X), _dtype_code(X), N, d, X.stride(0), _ptr(W),
                                  _ptr(b.float().contiguous()), D, _ptr(out), _dtype_code(out),
                                  _stream(X))
    _check("sls_feature_map_ex", st)
    return out


def feature_map_batched(X: torch.Tensor, W: torch.Tensor, b: torch.Tensor, rows: int,
                        live: Optional[torch.Tensor] = None, win: int = 0,
                        out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Features of the first `rows` rows of every prompt of a B x N x d bf16
    batch in one launch (Sec. 3.2, Eq. rff_map); with `live` (int32, B x nwin
    window flags, Sec. 3.6) only the row tiles of live windows are written.
    Returns B * rows x D float32."""
    _need_cuda(X, W, b)
    B, N, d = X.shape
    D = W.shape[0]
    assert X.stride(2) == 1 and X.stride(0) == N * X.stride(1)
    assert W.shape[1] == d and W.dtype == X.dtype and W.is_contiguous()
    if out is None:
        out = torch.empty((B * rows, D), dtype=torch.float32, device=X.device)
    nwin = 0
    lp = None
    if live is not None:
        live = live.to(device=X.device, dtype=torch.int32).contiguous()
        nwin = live.numel() // max(1, B)
        lp = _ptr(live)
    st = lib().sls_feature_map_batched(_ptr(X), B, rows, N, d, X.stride(1), _ptr(W),
                                       _ptr(b.float().contiguous()), D, _ptr(out), lp, nwin,
                                       win, _stream(X))
    _check("sls_feature_map_batched", st)
    return out


def feature_normalize(Phi: torch.Tensor):
    """The row-normalised operator of Sec. 3.2 in its symmetric form: the rows
    of Phi (N x D float32, in place) scaled by 1 / sqrt(s_i) with
    s = Phi (Phi^T 1).  Returns s (N float64)."""
    _need_cuda(Phi)
    assert Phi.dtype == torch.float32 and Phi.is_contiguous()
    N, D = Phi.shape
    s = torch.empty(N, dtype=torch.float64, device=Phi.device)
    L = lib()
    nbytes = L.sls_feature_normalize_workspace_size(N, D)
    ws = _workspace(max(nbytes, 256), Phi.device)
    _check("sls_feature_normalize",
           L.sls_feature_normalize(_ptr(Phi), N, D, _ptr(s), _ptr(ws), nbytes, _stream(Phi)))
    return s


def lanczos_topr(Phi: torch.Tensor, q1: torch.Tensor, r: int, tol: float = 1e-10):
    """Algorithm 2 on A(v) = Phi (Phi^T v), then Eigh(T) and U = Q V
    (Algorithm 1); Phi is float32 or bfloat16 (N x D).  Returns (theta[r]
    float64 descending, U[N, r] float32, r_eff[1] int32, alpha[r], beta[r])
    as device tensors."""
    _need_cuda(Phi, q1)
    Phi = Phi.contiguous()
    N, D = Phi.shape
    dev = Phi.device
    q1 = q1.to(device=dev, dtype=torch.float64).contiguous()
    theta = torch.empty(r, dtype=torch.float64, device=dev)
    U = torch.empty((N, r), dtype=torch.float32, device=dev)
    r_eff = torch.empty(1, dtype=torch.int32, device=dev)
    alpha = torch.empty(r, dtype=torch.float64, device=dev)
    beta = torch.empty(r, dtype=torch.float64, device=dev)
    L = lib()
    nbytes = L.sls_lanczos_workspace_size(N, D, r)
    if nbytes == 0:
        raise SLSError("sls_lanczos_workspace_size", 2, "unsupported shape")
    ws = _workspace(nbytes, dev)
    st = L.sls_lanczos_topr_ex(_ptr(Phi), _dtype_code(Phi), N, D, r, _ptr(q1), float(tol),
                               _ptr(theta), _ptr(U), _ptr(r_eff), _ptr(alpha), _ptr(beta),
                               _ptr(ws), ws.numel(), _stream(Phi))
    _check("sls_lanczos_topr_ex", st)
    _check_ws("sls_lanczos_topr_ex", ws)
    return theta, U, r_eff, alpha, beta


def lanczos_topr_batched(Phi: torch.Tensor, q1: torch.Tensor, r: int, row0, n, q1off=None,
                         tol: float = 1e-10):
    """Algorithm 2 and the Ritz pairs for several independent problems in one
    launch, with the plan the windowed backends use (Sec. 3.5-3.6): problem p
    owns rows row0[p] .. row0[p] + n[p] of Phi (float32 or bfloat16, rows x D)
    and starts from q1[q1off[p]:] (q1off defaults to row0).  Returns (theta
    [nprob, r] float64, U [rows, r] float32, r_eff [nprob] int32, alpha, beta)
    as device tensors."""
    _need_cuda(Phi, q1)
    Phi = Phi.contiguous()
    rows, D = Phi.shape
    dev = Phi.device
    row0_t = torch.as_tensor(row0, dtype=torch.int64).to(dev).contiguous()
    n_t = torch.as_tensor(n, dtype=torch.int32).to(dev).contiguous()
    nprob = int(n_t.numel())
    q1off_t = (torch.as_tensor(q1off, dtype=torch.int64).to(dev).contiguous()
               if q1off is not None else None)
    nmax = int(torch.as_tensor(n).max().item())
    q1 = q1.to(device=dev, dtype=torch.float64).contiguous()
    theta = torch.empty((nprob, r), dtype=torch.float64, device=dev)
    U = torch.zeros((rows, r), dtype=torch.float32, device=dev)
    r_eff = torch.empty(nprob, dtype=torch.int32, device=dev)
    alpha = torch.empty((nprob, r), dtype=torch.float64, device=dev)
    beta = torch.empty((nprob, r), dtype=torch.float64, device=dev)
    L = lib()
    nbytes = L.sls_lanczos_batched_workspace_size(rows, nmax, D, r, nprob)
    if nbytes == 0:
        raise SLSError("sls_lanczos_batched_workspace_size", 2, "unsupported shape")
    ws = _workspace(nbytes, dev)
    st = L.sls_lanczos_topr_batched(_ptr(Phi), _dtype_code(Phi), D, r, nprob, _ptr(row0_t),
                                    _ptr(n_t), _ptr(q1off_t), nmax, rows, _ptr(q1), float(tol),
                                    _ptr(theta), _ptr(U), _ptr(r_eff), _ptr(alpha),
                                    _ptr(beta), _ptr(ws), ws.numel(), _stream(Phi))
    _check("sls_lanczos_topr_batched", st)
    _check_ws("sls_lanczos_topr_batched", ws)
    return theta, U, r_eff, alpha, beta


def selftest_lanczos_giveup(Phi: torch.Tensor, q1: torch.Tensor, r: int):
    """The Lanczos kernel's failure path on a real problem (see
    sls_selftest_lanczos_giveup): returns (status word, theta, U, r_eff); the
    status is SLS_ERR_TIMEOUT = 5 and r_eff -1 when the kernel gave up as
    designed.  Takes about one second."""
    _need_cuda(Phi, q1)
    Phi = Phi.contiguous()
    N, D = Phi.shape
    dev = Phi.device
    q1 = q1.to(device=dev, dtype=torch.float64).contiguous()
    theta = torch.full((r,), 7.0, dtype=torch.float64, device=dev)
    U = torch.full((N, r), 7.0, dtype=torch.float32, device=dev)
    r_eff = torch.full((1,), 7, dtype=torch.int32, device=dev)
    L = lib()
    nbytes = L.sls_lanczos_workspace_size(N, D, r)
    ws = _workspace(nbytes, dev)
    st = L.sls_selftest_lanczos_giveup(_ptr(Phi), N, D, r, _ptr(q1), _ptr(theta), _ptr(U),
                                       _ptr(r_eff), _ptr(ws), ws.numel(), _stream(Phi))
    _check("sls_selftest_lanczos_giveup", st)
    status = int(L.sls_workspace_status(_ptr(ws), _stream(ws)))
    return status, theta, U, r_eff


def simhash(U: torch.Tensor, R: torch.Tensor, bits: int, k: Optional[int] = None,
            k_dev: Optional[torch.Tensor] = None) -> torch.Tensor:
    """SimHash codes of the rows of U (Sec. 3.3, Eq. simhash) against the
    first `bits` rows of R; returns N uint32 codes as an int32 tensor."""
    _need_cuda(U, R)
    N, ldu = U.shape[0], U.stride(0)
    k = U.shape[1] if k is None else k
    R = R.float().contiguous()
    codes = torch.empty(N, dtype=torch.int32, device=U.device)
    st = lib().sls_simhash(_ptr(U), N, k, ldu, _ptr(k_dev), _ptr(R), bits, R.stride(0),
                           _ptr(codes), _stream(U))
    _check("sls_simhash", st)
    return codes


def aggregate(X: torch.Tensor, codes: torch.Tensor, M_target: int, pos_scheme: int = POS_MAX,
              renorm: bool = True):
    """Clusters of equal codes, adjusted to exactly M_target groups, merged
    into macro-tokens ordered by position (Sec. 3.3-3.4).  Returns
    (Xt[M, d] float32, pos[M] int32, tok2macro[N] int32)."""
    _need_cuda(X, codes)
    N, d = X.shape
    dev = X.device
    Xt = torch.empty((M_target, d), dtype=torch.float32, device=dev)
    pos = torch.empty(M_target, dtype=torch.int32, device=dev)
    t2m = torch.empty(N, dtype=torch.int32, device=dev)
    L = lib()
    nbytes = L.sls_aggregate_workspace_size(N, d, M_target)
    if nbytes == 0:
        raise SLSError("sls_aggregate_workspace_size", 1, "invalid shape")
    ws = _workspace(nbytes, dev)
    st = L.sls_aggregate(_ptr(X), _dtype_code(X), N, d, X.stride(0), _ptr(codes.contiguous()),
                         M_target, pos_scheme, int(renorm), _ptr(Xt), _ptr(pos), _ptr(t2m),
                         _ptr(ws), ws.numel(), _stream(X))
    _check("sls_aggregate", st)
    _check_ws("sls_aggregate", ws)
    return Xt, pos, t2m


def output_count(cfg: Config, N: int) -> int:
    return int(lib().sls_output_count(ctypes.byref(cfg), N))


def compress_workspace_size(cfg: Config, B: int, N: int, d: int) -> int:
    return int(lib().sls_compress_workspace_size(ctypes.byref(cfg), B, N, d))


class Workspace:
    """A reusable device workspace for compress() (sized for one shape)."""

    def __init__(self, cfg: Config, B: int, N: int, d: int, device):
        self.nbytes = compress_workspace_size(cfg, B, N, d)
        if self.nbytes == 0:
            raise SLSError("sls_compress_workspace_size", 1, "invalid configuration")
        self.buf = _workspace(self.nbytes, device)


def _outputs(cfg: Config, B: int, N: int, d: int, dev, out):
    M = output_count(cfg, N)
    if M < 0:
        raise SLSError("sls_output_count", 1, "invalid configuration")
    if out is None:
        Xt = torch.empty((B, M, d), dtype=torch.float32, device=dev)
        pos = torch.empty((B, M), dtype=torch.int32, device=dev)
        t2m = torch.empty((B, N), dtype=torch.int32, device=dev)
    else:
        Xt, pos, t2m = out
    nwin = max(1, B * ((N + max(1, cfg.window) - 1) // max(1, cfg.window)))
    r_eff = torch.zeros(nwin, dtype=torch.int32, device=dev)
    route = torch.zeros(nwin, dtype=torch.int32, device=dev)
    return M, Xt, pos, t2m, r_eff, route


def _params(cfg: Config, M: int, N: int, B: int, batched: bool, dev, W, b, R, q1):
    """sls_params_t for the spectral backends (None for chunk or identity),
    and the contiguous tensors it points into (kept alive by the caller)."""
    if cfg.backend == BACKEND_CHUNK or M == N:
        return None, []
    if W is None or b is None or R is None or q1 is None:
        raise ValueError("the spectral backends need W, b, R and q1")
    Wc = W.contiguous()
    bc = b.float().contiguous()
    Rc = R.float().contiguous()
    qc = q1.to(device=dev, dtype=torch.float64).contiguous()
    q1_stride = qc.numel() // B if batched else 0
    params = _Params(Wc.data_ptr(), bc.data_ptr(), Rc.data_ptr(), Rc.shape[0], Rc.stride(0),
                     qc.data_ptr(), q1_stride)
    return params, [Wc, bc, Rc, qc]


def compress(X: torch.Tensor, cfg: Config, W: Optional[torch.Tensor] = None,
             b: Optional[torch.Tensor] = None, R: Optional[torch.Tensor] = None,
             q1: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
             out=None):
    """The whole compression pass (Algorithm 1 with the backends of Sec. 3.5
    and 3.6).  X is N x d or B x N x d (float32 or bfloat16).  Returns
    (Xt, pos, tok2macro, r_eff, route); Xt is [B,] M x d float32."""
    _need_cuda(X)
    batched = X.dim() == 3
    X3 = X if batched else X.unsqueeze(0)
    B, N, d = X3.shape
    assert X3.stride(2) == 1 and X3.stride(0) == N * X3.stride(1)
    dev = X.device
    M, Xt, pos, t2m, r_eff, route = _outputs(cfg, B, N, d, dev, out)
    if workspace is None:
        workspace = Workspace(cfg, B, N, d, dev)
    params, keep = _params(cfg, M, N, B, batched, dev, W, b, R, q1)
    st = lib().sls_compress(ctypes.byref(cfg), _ptr(X3), _dtype_code(X3), B, N, d,
                            X3.stride(1), ctypes.byref(params) if params is not None else None,
                            _ptr(Xt), _ptr(pos), _ptr(t2m), _ptr(r_eff), _ptr(route),
                            _ptr(workspace.buf), workspace.nbytes, _stream(X3))
    _check("sls_compress", st)
    _check_ws("sls_compress", workspace.buf)
    del keep
    if not batched:
        return Xt[0], pos[0], t2m[0], r_eff, route
    return Xt, pos, t2m, r_eff, route


def embed_gather(table: torch.Tensor, ids: torch.Tensor, out: Optional[torch.Tensor] = None,
                 bad: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Input embeddings X = table[ids] (Sec. 3.1): table is V x d (float32 or
    bfloat16), ids any shape of int32 token ids; returns ids.shape + (d,) in
    the table's dtype.  Rows of out-of-range ids are zero; `bad` (one int32,
    optional) receives their count."""
    _need_cuda(table, ids, out, bad)
    V, d = table.shape
    assert table.stride(1) == 1
    ids_c = ids.to(dtype=torch.int32).contiguous()
    N = ids_c.numel()
    if out is None:
        out = torch.empty(tuple(ids.shape) + (d,), dtype=table.dtype, device=table.device)
    assert out.dtype == table.dtype and out.is_contiguous()
    st = lib().sls_embed_gather(_ptr(table), _dtype_code(table), V, d, table.stride(0),
                                _ptr(ids_c), N, _ptr(out), d, _ptr(bad), _stream(table))
    _check("sls_embed_gather", st)
    return out


def compress_tokens_workspace_size(cfg: Config, dtype: torch.dtype, B: int, N: int,
                                   d: int) -> int:
    code = SLS_BF16 if dtype == torch.bfloat16 else SLS_F32
    return int(lib().sls_compress_tokens_workspace_size(ctypes.byref(cfg), code, B, N, d))


class TokensWorkspace:
    """A reusable device workspace for compress_tokens() (one shape)."""

    def __init__(self, cfg: Config, dtype: torch.dtype, B: int, N: int, d: int, device):
        self.nbytes = compress_tokens_workspace_size(cfg, dtype, B, N, d)
        if self.nbytes == 0:
            raise SLSError("sls_compress_tokens_workspace_size", 1, "invalid configuration")
        self.buf = _workspace(self.nbytes, device)


def compress_tokens(ids: torch.Tensor, table: torch.Tensor, cfg: Config,
                    W: Optional[torch.Tensor] = None, b: Optional[torch.Tensor] = None,
                    R: Optional[torch.Tensor] = None, q1: Optional[torch.Tensor] = None,
                    workspace: Optional[TokensWorkspace] = None, out=None,
                    bad: Optional[torch.Tensor] = None):
    """compress() from token ids (N or B x N int32) and the model's input
    embedding table (V x d): the lookup X = table[ids] (Sec. 3.1) and the
    compression pass in one call.  Returns what compress() returns."""
    _need_cuda(ids, table, bad)
    batched = ids.dim() == 2
    ids2 = (ids if batched else ids.view(1, -1)).to(dtype=torch.int32).contiguous()
    B, N = ids2.shape
    V, d = table.shape
    assert table.stride(1) == 1
    dev = table.device
    M, Xt, pos, t2m, r_eff, route = _outputs(cfg, B, N, d, dev, out)
    if workspace is None:
        workspace = TokensWorkspace(cfg, table.dtype, B, N, d, dev)
    params, keep = _params(cfg, M, N, B, batched, dev, W, b, R, q1)
    st = lib().sls_compress_tokens(ctypes.byref(cfg), _ptr(table), _dtype_code(table), V, d,
                                   table.stride(0), _ptr(ids2), B, N,
                                   ctypes.byref(params) if params is not None else None,
                                   _ptr(Xt), _ptr(pos), _ptr(t2m), _ptr(r_eff), _ptr(route),
                                   _ptr(bad), _ptr(workspace.buf), workspace.nbytes,
                                   _stream(table))
    _check("sls_compress_tokens", st)
    del keep
    if not batched:
        return Xt[0], pos[0], t2m[0], r_eff, route
    return Xt, pos, t2m, r_eff, route


def set_phase_events(events) -> None:
    """Record torch.cuda.Event pairs around the phases of compress() (see
    sls_set_phase_events); None switches timing off."""
    if events is None:
        _check("sls_set_phase_events", lib().sls_set_phase_events(None, 0))
        return
    arr = (ctypes.c_void_p * len(events))(*[e.cuda_event for e in events])
    _check("sls_set_phase_events", lib().sls_set_phase_events(arr, len(events)))


def launch_count() -> int:
    """Kernels launched by libsls in this process so far."""
    return int(lib().sls_launch_count())


def selftest_wait_limit(which: int, device="cuda") -> int:
    """Run the self-test of the device-side wait limits (which = 0: an
    mbarrier nothing completes; 1: a group barrier one CTA never reaches) and
    return the status it leaves (SLS_ERR_TIMEOUT = 5 when the wait gave up as
    designed).  Takes about one second."""
    ws = _workspace(512, device)
    st = lib().sls_selftest_wait_limit(int(which), _ptr(ws), ws.numel(),
                                       _stream(ws))
    _check("sls_selftest_wait_limit", st)
    return int(lib().sls_workspace_status(_ptr(ws), _stream(ws)))


def workspace_status(workspace: Workspace) -> int:
    """Device status word of a compress workspace (0 = ok, 5 = timeout)."""
    return int(lib().sls_workspace_status(_ptr(workspace.buf),
                                          _stream(workspace.buf)))

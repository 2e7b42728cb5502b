"""sls_lanczos_topr_noalloc: the Lanczos call for callers that may not
allocate device memory (its scratch is a fixed device array inside the
library).  Called through the C ABI, its results must match the workspace
entry point sls_lanczos_topr within the parity tolerances, on two calls in a
row with different problems (the shared scratch keeps the previous call's
contents)."""
import ctypes

import numpy as np
import pytest
import scipy.linalg
import torch

import oracle as O
import workloads as WL

pytestmark = pytest.mark.gpu


def _problem(N, D, seed):
    g = np.random.default_rng(seed)
    X = g.standard_normal((N, 24)) / np.sqrt(24)
    W = g.standard_normal((D, 24)) * 24 ** -0.25
    b = g.random(D) * 2 * np.pi
    return O.rff_features(X, W, b).astype(np.float32), g.standard_normal(N)


def test_noalloc_matches_workspace_entry_point():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as sls
    L = sls.lib()
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for N, D, r, seed in [(3000, 512, 32, 1), (700, 256, 16, 2)]:
        phi, q1 = _problem(N, D, seed)
        Phi = torch.from_numpy(phi).cuda()
        Q1 = torch.from_numpy(q1).cuda()
        th_ref, U_ref, k_ref, _, _ = sls.lanczos_topr(Phi, Q1, r)
        theta = torch.empty(r, dtype=torch.float64, device="cuda")
        U = torch.empty((N, r), dtype=torch.float32, device="cuda")
        k = torch.empty(1, dtype=torch.int32, device="cuda")
        st = L.sls_lanczos_topr_noalloc(ctypes.c_void_p(Phi.data_ptr()), N, D, r,
                                        ctypes.c_void_p(Q1.data_ptr()), 1e-10,
                                        ctypes.c_void_p(theta.data_ptr()),
                                        ctypes.c_void_p(U.data_ptr()),
                                        ctypes.c_void_p(k.data_ptr()), None, None, s)
        assert st == 0, L.sls_status_string(st)
        torch.cuda.synchronize()
        kk = int(k.item())
        assert kk == int(k_ref.item()) and kk > 0
        a = theta.cpu().numpy()[:kk]
        b = th_ref.cpu().numpy()[:kk]
        assert np.all(np.abs(a - b) <= 1e-4 * np.abs(b) + 1e-12 * abs(b[0]))
        ang = scipy.linalg.subspace_angles(U.cpu().numpy()[:, :kk].astype(np.float64),
                                           U_ref.cpu().numpy()[:, :kk].astype(np.float64))
        assert np.max(ang) <= 1e-3
    # sizes past the fixed scratch are refused with a clear error, before
    # anything is enqueued: real buffers of a problem whose workspace is just
    # over the limit (the basis alone is 41 MB), r_eff left untouched
    N, D, r = 40000, 256, 128
    need = L.sls_lanczos_workspace_size(N, D, r)
    assert (32 << 20) < need < (64 << 20)
    phi, q1 = _problem(N, D, 3)
    Phi = torch.from_numpy(phi).cuda()
    Q1 = torch.from_numpy(q1).cuda()
    theta = torch.zeros(r, dtype=torch.float64, device="cuda")
    U = torch.zeros((N, r), dtype=torch.float32, device="cuda")
    k = torch.full((1,), 12345, dtype=torch.int32, device="cuda")
    st = L.sls_lanczos_topr_noalloc(ctypes.c_void_p(Phi.data_ptr()), N, D, r,
                                    ctypes.c_void_p(Q1.data_ptr()), 1e-10,
                                    ctypes.c_void_p(theta.data_ptr()),
                                    ctypes.c_void_p(U.data_ptr()),
                                    ctypes.c_void_p(k.data_ptr()), None, None, s)
    assert st == 3
    torch.cuda.synchronize()
    assert int(k.item()) == 12345

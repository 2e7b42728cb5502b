"""The debug build of the library (libsls_debug.so, compiled with
-DSLS_DEBUG) as the stand-in for a memory checker: every workspace region
it carves is followed by a guard band that is filled when a call starts and
checked when it ends, and selected device-side accesses (row indices of the
Lanczos kernel, member rows of the aggregation) are guarded, so that an
access outside its range is skipped and reported as SLS_ERR_BOUNDS in the
workspace status word instead of faulting.

Two checks: the self-test plants both kinds of mistake (a write into a guard
band, inside the caller's own buffer, and a guarded out-of-range write) and
must see SLS_ERR_BOUNDS; and the parity cases of the stage and batched tests
run again on the debug build with the status word read after every call
(SLS_CHECK_STATUS=1), which must stay SLS_OK while the results still match
the oracle."""
import ctypes
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SLS_OK, SLS_ERR_UNSUPPORTED, SLS_ERR_BOUNDS = 0, 2, 6


@pytest.fixture(scope="module")
def debug_lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as sls
    from paper_2607_19368_gb300 import build
    path = sls.debug_lib_path()
    if not os.path.exists(path):
        build.build(debug=True)
    L = ctypes.CDLL(path)
    L.sls_debug_selftest.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t,
                                     ctypes.c_void_p]
    L.sls_workspace_status.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    return L


@pytest.mark.parametrize("which", [0, 1])
def test_debug_checks_catch_planted_mistakes(debug_lib, which):
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = debug_lib.sls_debug_selftest(which, ctypes.c_void_p(ws.data_ptr()), ws.numel(), s)
    assert st == SLS_OK
    assert debug_lib.sls_workspace_status(ctypes.c_void_p(ws.data_ptr()), s) == SLS_ERR_BOUNDS


def test_ordinary_build_has_no_checks():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as sls
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert sls.lib().sls_debug_selftest(0, ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                                        s) == SLS_ERR_UNSUPPORTED


def test_parity_cases_clean_under_debug_build(debug_lib):
    import paper_2607_19368_gb300 as sls
    env = dict(os.environ, SLS_LIBRARY=sls.debug_lib_path(), SLS_CHECK_STATUS="1")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_gpu_parity.py", "tests/test_gpu_batched.py"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    tail = "\n".join((r.stdout + r.stderr).strip().splitlines()[-15:])
    assert r.returncode == 0, tail
    assert " passed" in tail and "failed" not in tail, tail

"""The C ABI: the library builds for sm_103a, loads without a GPU and exports
every entry point declared in include/sls.h; host-side argument checks and
the output-count arithmetic need no GPU either."""
import ctypes
import os
import re

import pytest
import torch

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sls.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w \*]*?\b(sls_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_19368_gb300 import build
    path = build.build()
    import paper_2607_19368_gb300 as sls
    return sls.lib()


def test_header_declares_the_five_calls():
    names = declared_functions()
    for n in ("sls_feature_map", "sls_lanczos_topr", "sls_simhash", "sls_aggregate",
              "sls_compress"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    import paper_2607_19368_gb300 as sls
    names = declared_functions()
    assert set(names) == set(sls.EXPORTED), (set(names) ^ set(sls.EXPORTED))
    for n in names:
        assert hasattr(lib, n), n


def test_host_side_errors_and_counts(lib):
    import paper_2607_19368_gb300 as sls
    assert lib.sls_version() >= 100
    assert lib.sls_status_string(5).decode().startswith("device wait")
    # argument errors are detected before any CUDA call
    assert lib.sls_feature_map(None, 0, 4, 8, 8, None, None, 6, None, None) == 1  # D % 4
    assert lib.sls_simhash(None, 4, 4, 4, None, None, 33, 4, None, None) == 1     # bits > 32
    # batched features: prompt stride below the row count; windows not covering the rows
    assert lib.sls_feature_map_batched(None, 2, 10, 5, 8, 8, None, None, 256, None, None, 0, 0,
                                       None) == 1
    assert lib.sls_feature_map_batched(None, 2, 10, 10, 8, 8, None, None, 256, None,
                                       ctypes.c_void_p(16), 2, 4, None) == 1
    assert lib.sls_lanczos_topr(None, 4, 8, 0, None, 1e-10, None, None, None, None, None,
                                None, 0, None) == 1                               # r = 0
    assert lib.sls_lanczos_workspace_size(1000, 256, 16) > 0
    # batched Lanczos: no problems; a NULL problem table
    assert lib.sls_lanczos_topr_batched(None, 0, 256, 16, 0, None, None, None, 100, 100, None,
                                        1e-10, None, None, None, None, None, None, 0, None) == 1
    assert lib.sls_lanczos_topr_batched(ctypes.c_void_p(256), 0, 256, 16, 2, None, None, None,
                                        100, 200, ctypes.c_void_p(256), 1e-10,
                                        ctypes.c_void_p(256), ctypes.c_void_p(256), None, None,
                                        None, None, 0, None) == 1
    assert lib.sls_lanczos_batched_workspace_size(200, 100, 256, 16, 2) > 0
    # the give-up self-test has no barrier to fail in the one-warp window kernel
    assert lib.sls_selftest_lanczos_giveup(ctypes.c_void_p(256), 20, 256, 16,
                                           ctypes.c_void_p(256), ctypes.c_void_p(256),
                                           ctypes.c_void_p(256), ctypes.c_void_p(256), None,
                                           0, None) == 2
    # embedding lookup: table stride below d, unknown dtype, missing ids
    assert lib.sls_embed_gather(None, 1, 10, 8, 4, None, 4, None, 8, None, None) == 1
    assert lib.sls_embed_gather(None, 7, 10, 8, 8, None, 4, None, 8, None, None) == 1
    assert lib.sls_embed_gather(ctypes.c_void_p(16), 1, 10, 8, 8, None, 4, ctypes.c_void_p(16),
                                8, None, None) == 1
    assert lib.sls_embed_gather(None, 1, 10, 8, 8, None, 0, None, 8, None, None) == 0  # N = 0
    # bf16 storage of Phi with the normalised operator: unsupported, before any CUDA call
    bad = sls.Config.make(rho=4.0, D=256, r=8, normalize=1, phi_dtype=sls.SLS_BF16)
    assert sls.output_count(bad, 100) == -1
    assert lib.sls_compress_tokens(ctypes.byref(bad), ctypes.c_void_p(256), 1, 10, 64, 64,
                                   ctypes.c_void_p(256), 1, 100, None, None, None, None, None,
                                   None, None, None, 0, None) == 2
    assert lib.sls_selftest_wait_limit(2, None, 0, None) == 1          # which out of range
    cfg = sls.Config.make(rho=16.0, D=2048, r=64, bits=16)
    assert (sls.compress_tokens_workspace_size(cfg, torch.bfloat16, 1, 32768, 3584)
            >= sls.compress_workspace_size(cfg, 1, 32768, 3584) + 32768 * 3584 * 2)
    # output counts agree with the oracle's target count (Sec. 3.3) and identity
    for N, rho, pf, pl in [(512, 4.0, 0, 12), (16384, 16.0, 0, 12), (100, 1.0, 0, 12),
                           (10, 4.0, 3, 20), (1000, 3.0, 5, 7)]:
        cfg = sls.Config.make(rho=rho, preserve_first=pf, preserve_last=pl)
        Nc = N - min(pf, N) - min(pl, N - min(pf, N))
        want = N if (rho <= 1 or Nc <= 0) else min(pf, N) + O.target_count(Nc, rho) + min(pl, N - min(pf, N))
        assert sls.output_count(cfg, N) == want
    cfg = sls.Config.make(backend=sls.BACKEND_CHUNK, rho=2.5, preserve_last=0)
    assert sls.output_count(cfg, 101) == -(-101 // round(2.5))
    assert sls.compress_workspace_size(sls.Config.make(rho=16.0, D=2048, r=64, bits=16),
                                       1, 32768, 3584) > 32768 * 2048 * 4

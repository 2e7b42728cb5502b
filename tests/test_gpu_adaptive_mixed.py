"""The adaptive router (Sec. 3.6) at the adaptive workload's real shape --
windows of 2048 tokens, d = 4096 bf16, D = 1024, r = 32 -- on prompts of the
mixed generator (coherent windows among low-redundancy ones), so that one
call routes windows both ways at rho = 4 and 8.  The routes must be the
oracle's; the chunk windows' macro-tokens, positions and token maps the
oracle's exactly (embeddings to 1e-4); the spectral windows' groups must
satisfy the pass invariants, with their macro embeddings and positions
recomputed by the oracle from the GPU's own groups."""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import to_torch_x
from tests.test_gpu_parity import EMB_TOL, _check_pass

pytestmark = pytest.mark.gpu

PROMPTS = (1, 9)  # one coherent window of three, and two of three


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


@pytest.fixture(scope="module")
def mixed():
    w = WL.scaled(WL.WORKLOADS["adaptive_mixed"], N=6144, batch=len(PROMPTS))
    X = np.stack([WL.make_prompt(w, index=i).X for i in PROMPTS])
    prm = WL.make_params(w.D, w.d, w.r, 32, len(PROMPTS) * w.N, "bf16")
    return w, X, prm


@pytest.mark.parametrize("rho", [4.0, 8.0])
def test_adaptive_router_mixed_at_workload_shape(sls, mixed, rho):
    w, X, prm = mixed
    B, N = X.shape[0], w.N
    pl = w.preserve_last
    cfg = sls.Config.make(backend=sls.BACKEND_ADAPTIVE, rho=rho, D=w.D, r=w.r, window=w.window,
                          preserve_last=pl)
    Xt, pos, t2m, r_eff, route = sls.compress(to_torch_x(X, "bf16"), cfg,
                                              to_torch_x(prm.W, "bf16"),
                                              torch.from_numpy(prm.b).cuda(),
                                              torch.from_numpy(prm.R).cuda(),
                                              torch.from_numpy(prm.q1).cuda())
    torch.cuda.synchronize()
    M = sls.output_count(cfg, N)
    bounds = O.window_bounds(N - pl, w.window)
    route = route.cpu().numpy()[:B * len(bounds)].reshape(B, len(bounds))
    r_eff = r_eff.cpu().numpy()[:B * len(bounds)].reshape(B, len(bounds))
    n_spec = 0
    for i in range(B):
        x64 = WL.bf16_bits_to_f32(X[i]).astype(np.float64)
        res = O.compress_adaptive(x64, prm.w_f64(), prm.b, prm.R, prm.q1[i * N:(i + 1) * N],
                                  O.CompressConfig(rho=rho, D=w.D, r=w.r, window=w.window,
                                                   preserve_last=pl))
        coherent = {a for a, _, _ in WL.coherent_windows(w, index=PROMPTS[i])}
        for k, ((s_, e_), sp) in enumerate(zip(bounds, res.info["spectral"])):
            assert route[i, k] == int(sp)
            assert bool(sp) == (s_ in coherent)  # the generator's coherent windows
            assert r_eff[i, k] == (w.r if sp else 0)
        n_spec += int(route[i].sum())
        _check_pass(sls, x64, Xt[i].cpu().numpy(), pos[i].cpu().numpy(), t2m[i].cpu().numpy(),
                    M, 0, pl)
        t = t2m[i].cpu().numpy()
        for k, (s_, e_) in enumerate(bounds):
            if not route[i, k]:
                assert np.array_equal(t[s_:e_], res.tok2macro[s_:e_])
                ms = np.unique(res.tok2macro[s_:e_])
                assert np.array_equal(pos[i].cpu().numpy()[ms], res.pos[ms])
                assert np.max(np.abs(Xt[i].cpu().numpy()[ms] - res.Xt[ms])) <= EMB_TOL
    assert 0 < n_spec < B * len(bounds)

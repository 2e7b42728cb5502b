"""The step before the pass (Sec. 3.1, Fig. 1): input embeddings looked up by
token id on the GPU, bit for bit against the oracle's lookup, and the whole
pass from token ids against the pass from the oracle's X."""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests.gpu_util import to_torch_x

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19368_gb300 as m
    m.lib()
    return m


def _table(rng, V, ld, dtype):
    """A V x ld table of random bits (float32 values, or bf16 patterns); only
    the first d columns are the embeddings when ld > d."""
    if dtype == "bf16":
        return WL.f32_to_bf16_bits(rng.standard_normal((V, ld)).astype(np.float32))
    return rng.standard_normal((V, ld)).astype(np.float32)


def _bits(a):
    a = np.ascontiguousarray(a)
    return a.view(np.uint16) if a.dtype.itemsize == 2 else a.view(np.uint32)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("V,d,ld,N", [(1000, 3584, 3584, 4099),   # 16-byte rows
                                       (50, 24, 24, 333),          # 16-byte rows, short
                                       (77, 13, 13, 257),          # element copies
                                       (64, 40, 48, 100),          # strided table
                                       (5, 8, 8, 1),               # one token
                                       (5, 8, 8, 0)])              # empty prompt
def test_embed_gather_bit_exact(sls, dtype, V, d, ld, N):
    rng = np.random.default_rng(V * 7 + d)
    tab = _table(rng, V, ld, dtype)
    ids = rng.integers(-2, V + 2, size=N).astype(np.int32)    # a few out of range
    if N > 2:
        ids[:2] = [0, V - 1]
    want = O.embed_lookup(np.ascontiguousarray(tab[:, :d]), ids)
    t = to_torch_x(tab, dtype)[:, :d]
    bad = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    X = sls.embed_gather(t, torch.from_numpy(ids).cuda(), bad=bad)
    torch.cuda.synchronize()
    assert tuple(X.shape) == (N, d)
    got = X.view(torch.int16).cpu().numpy() if dtype == "bf16" else X.cpu().numpy()
    assert np.array_equal(_bits(got), _bits(want))
    assert int(bad.item()) == int(np.sum((ids < 0) | (ids >= V)))


def test_embed_gather_batched_ids(sls):
    rng = np.random.default_rng(3)
    tab = _table(rng, 300, 64, "bf16")
    ids = rng.integers(0, 300, size=(4, 129)).astype(np.int32)
    X = sls.embed_gather(to_torch_x(tab, "bf16"), torch.from_numpy(ids).cuda())
    assert tuple(X.shape) == (4, 129, 64)
    want = O.embed_lookup(tab, ids.reshape(-1)).reshape(4, 129, 64)
    assert np.array_equal(X.view(torch.int16).cpu().numpy().view(np.uint16), want)


def _vocab_table(w):
    """The generator's full vocabulary (bf16 bits or float32), V x d."""
    rows = WL.vocab_rows(WL.DATA_SEED, np.arange(w.V), w.d).astype(np.float32)
    return WL.f32_to_bf16_bits(rows) if w.dtype == "bf16" else rows


@pytest.mark.parametrize("backend", ["global", "local"])
def test_compress_tokens_equals_compress_of_oracle_lookup(sls, backend):
    """The pass from token ids is the pass from X = E[ids] (X computed by the
    oracle's lookup), output for output: the lookup adds nothing else."""
    w = WL.scaled(WL.WORKLOADS["qwen7b"], N=1500, d=256, V=700, D=256, r=16, bits=10, rho=8.0)
    ids = WL.prompt_ids(w).astype(np.int32)
    tab = _vocab_table(w)
    X = O.embed_lookup(tab, ids)
    prm = WL.params_for(w)
    kw = dict(backend=sls.BACKEND_GLOBAL, rho=w.rho, D=w.D, r=w.r, bits=w.bits)
    if backend == "local":
        kw.update(backend=sls.BACKEND_LOCAL, window=16, bits=0, r=8)
    cfg = sls.Config.make(**kw)
    args = (to_torch_x(prm.W, w.dtype), torch.from_numpy(prm.b).cuda(),
            torch.from_numpy(prm.R).cuda(), torch.from_numpy(prm.q1).cuda())
    ref = sls.compress(to_torch_x(X, w.dtype), cfg, *args)
    bad = torch.zeros(1, dtype=torch.int32, device="cuda")
    got = sls.compress_tokens(torch.from_numpy(ids).cuda(), to_torch_x(tab, w.dtype), cfg,
                              *args, bad=bad)
    torch.cuda.synchronize()
    assert int(bad.item()) == 0
    for a, b in zip(ref, got):
        assert torch.equal(a, b)


def test_compress_tokens_batched_and_identity(sls):
    w = WL.scaled(WL.WORKLOADS["mistral7b"], N=600, d=64, V=500, D=256, r=8, bits=8, rho=4.0)
    tab = _vocab_table(w)
    ids = np.stack([WL.prompt_ids(w, index=k) for k in range(3)]).astype(np.int32)
    prm = WL.make_params(w.D, w.d, w.r, 32, 3 * w.N, w.dtype)
    args = (to_torch_x(prm.W, w.dtype), torch.from_numpy(prm.b).cuda(),
            torch.from_numpy(prm.R).cuda(), torch.from_numpy(prm.q1).cuda())
    X = O.embed_lookup(tab, ids.reshape(-1)).reshape(3, w.N, w.d)
    cfg = sls.Config.make(backend=sls.BACKEND_ADAPTIVE, rho=4.0, D=w.D, r=w.r, window=200)
    ref = sls.compress(to_torch_x(X, w.dtype), cfg, *args)
    got = sls.compress_tokens(torch.from_numpy(ids).cuda(), to_torch_x(tab, w.dtype), cfg, *args)
    for a, b in zip(ref, got):
        assert torch.equal(a, b)
    # rho <= 1: the identity, i.e. the looked-up embeddings themselves
    cfg1 = sls.Config.make(rho=1.0)
    Xt, pos, t2m, _, _ = sls.compress_tokens(torch.from_numpy(ids[0]).cuda(),
                                             to_torch_x(tab, w.dtype), cfg1)
    want = WL.bf16_bits_to_f32(X[0]) if w.dtype == "bf16" else X[0]
    assert np.array_equal(Xt.cpu().numpy(), want)
    assert np.array_equal(pos.cpu().numpy(), np.arange(w.N))

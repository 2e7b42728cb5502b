"""Benchmark of the Spectral-LSH compression pass on GB300.

One step = one sls_compress call (features, Lanczos, Ritz vectors, SimHash,
clusters/adjust/order, macro-token aggregation) over one synthetic prompt of
the Qwen2.5-7B-shaped workload: N = 32768 tokens, d = 3584 bf16 embeddings,
D = 2048 RFF features, r = 64 Lanczos steps, b = 16 SimHash bits, rho = 16,
last 12 tokens preserved, global backend.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]
                  [--workload qwen7b|qwen14b|mistral7b|adaptive|local] [--rho R]

--workload qwen14b (N = 131072, d = 5120) and mistral7b (N = 8192, d = 4096)
time the other single-prompt shapes; --workload adaptive_mixed times the same
batch shape with about half of the windows coherent, so that the router
sends windows both ways at rho = 4 and 8; --workload adaptive times the windowed
batch: 64 prompts of N = 16384, d = 4096 bf16 (duplication 0.6 p / 63 for
prompt p), windows of 2048 routed to the chunk or the spectral chain, D = 1024,
r = 32, bits from the window budget, rho from --rho (default 8); --workload
local times local LSH (Spectral-LSH inside every window of 16 tokens) on the
Qwen2.5-7B-shaped prompt at the paper's defaults D = 256, r = 16, rho = 8.

The prompt (235 MB of embeddings) and the feature matrix (268 MB) are both
larger than the 129 MB L2, so no extra flush runs between steps.  With
--gpus N > 1 (torchrun, one rank per GPU) every rank compresses its own
prompt: independent replicas, no collective on the data path (weak scaling).
--impl reference times the CPU oracle (numpy float64) on a bounded sample of
the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tokens compressed/s at N=32k, rho=16 (1 GB300); Lanczos matvec HBM GB/s vs peak"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default="qwen7b",
                    choices=["qwen7b", "qwen14b", "mistral7b", "adaptive", "adaptive_mixed",
                             "local"])
    ap.add_argument("--rho", type=float, default=None,
                    help="compression ratio (default: the workload's)")
    ap.add_argument("--normalize", action="store_true",
                    help="row-normalised operator (the paper's untested Sec. 3.2 variant)")
    ap.add_argument("--phi", default="f32", choices=["f32", "bf16"],
                    help="storage of the feature matrix (bf16: opt-in half-size Phi)")
    ap.add_argument("--cpu-sample", type=int, default=4096,
                    help="tokens of the prompt the CPU oracle compresses per baseline step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the other workloads timed after the qwen7b headline")
    ap.add_argument("--sweep-steps", type=int, default=20)
    ap.add_argument("--ref-sample", type=int, default=1024,
                    help="tokens the oracle compresses per step of --impl reference")
    return ap.parse_args()


def workload(name):
    import workloads as WL
    return WL.WORKLOADS[name]


def config_dict(w, rho, extra=None):
    if w.backend == "local":
        d = {"workload": f"{w.name}: qwen7b-shaped prompt N={w.N} d={w.d} bf16, local LSH "
                         f"with windows of {w.window}, D={w.D} r={w.r} b=auto rho={rho:g} "
                         f"preserve_last={w.preserve_last}",
             "window": w.window,
             "l2": (f"inputs larger than L2 (X {w.N * w.d * 2 / 1e6:.0f} MB per step), "
                    f"no flush")}
    elif w.batch > 1:
        mix = (f", each window coherent (rows 0.8 t + 0.6 e_i) with probability "
               f"{w.coherent_frac:g}" if w.coherent_frac > 0 else "")
        d = {"workload": f"{w.name}: {w.batch} prompts of N={w.N} d={w.d} bf16, windows of "
                         f"{w.window}{mix}, D={w.D} r={w.r} b=auto rho={rho:g} "
                         f"preserve_last={w.preserve_last}, adaptive backend",
             "B": w.batch, "window": w.window,
             "l2": (f"inputs larger than L2 (X {w.batch * w.N * w.d * 2 / 1e9:.1f} GB per "
                    f"step), no flush")}
    else:
        d = {"workload": f"{w.name}-shaped prompt: N={w.N} d={w.d} bf16, D={w.D} r={w.r} "
                         f"b={w.bits} rho={rho:g} preserve_last={w.preserve_last}, "
                         f"global backend",
             "l2": (f"inputs larger than L2 (X {w.N * w.d * 2 / 1e6:.0f} MB and Phi "
                    f"{w.N * w.D * 4 / 1e6:.0f} MB per step), no flush")}
    d.update({"N": w.N, "d": w.d, "D": w.D, "r": w.r, "bits": w.bits, "rho": rho})
    if extra:
        d.update(extra)
    return d


# Revision of the persistent Lanczos kernel whose DRAM counters are recorded in
# profiles/lanczos_traffic.json; bumped with every change of the kernel, so a
# stale capture reads as "traffic": null.
LANCZOS_KERNEL_REV = "fused-pass/13"


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class Clocks:
    """nvidia-smi sampler running during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.p = None
        try:
            self.p = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", bus_id],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        out, _ = self.p.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "samples": len(sm),
                "reasons": sorted(reasons)}


def max_over_ranks(values, world, device):
    """The largest of each timing over all ranks (the slowest rank sets the
    job's time); the identity on one rank."""
    import torch
    t = torch.tensor(values, dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.tolist()]


def lanczos_one_pass_bytes(n_tokens, D, r, esz=4):
    """Per launch: what one fused pass per step has to move, one sweep over
    Phi per step (r D esz bytes per token) plus the same basis traffic."""
    return n_tokens * (esz * r * D + 16 * r * (r + 1))


def lanczos_algorithmic_bytes(n_tokens, D, r, esz=4):
    """Per launch: two sweeps over Phi per step (2 r D esz bytes per token:
    8 r D for float32 Phi, 4 r D for bf16) plus the double-float basis
    traffic of the two Gram-Schmidt passes (16 r (r + 1) bytes per token)."""
    return n_tokens * (2 * esz * r * D + 16 * r * (r + 1))


def windowed(w):
    return w.backend in ("adaptive", "local")


def window_lengths(w):
    """Lengths of the windows over one prompt's compressible region
    (consecutive windows, the last one shorter)."""
    nc = w.N - w.preserve_first - w.preserve_last
    return [min(w.window, nc - s) for s in range(0, nc, w.window)]


def oracle_config(w, rho):
    import oracle as O
    return O.CompressConfig(rho=rho, D=w.D, r=w.r, bits=w.bits,
                            preserve_first=w.preserve_first, preserve_last=w.preserve_last,
                            window=w.window if windowed(w) else 2048)


def cpu_oracle_step(w, rho, X64, prm, n):
    """One oracle compression of the first n tokens of a prompt (global
    backend, or the windowed backend of the workload)."""
    import oracle as O
    cfg = oracle_config(w, rho)
    t = time.perf_counter()
    if w.backend == "adaptive":
        O.compress_adaptive(X64[:n], prm.w_f64(), prm.b, prm.R, prm.q1[:n], cfg)
    elif w.backend == "local":
        O.compress_local(X64[:n], prm.w_f64(), prm.b, prm.R, prm.q1[:n], cfg)
    else:
        O.compress_global(X64[:n], prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
    return time.perf_counter() - t


def sample_prompt(w):
    """The prompt the CPU oracle samples: the only prompt of a single-prompt
    workload, the middle prompt of the adaptive batch."""
    import workloads as WL
    if w.batch > 1:
        i = w.batch // 2
        return WL.make_prompt(w, index=i, dup_frac=prompt_dup(w, i)), i
    return WL.make_prompt(w), 0


def prompt_dup(w, i):
    """Copied-span fraction of prompt i of a batch: varied over the prompts of
    the adaptive workload, the workload's own otherwise."""
    import workloads as WL
    return WL.adaptive_dup_frac(i, w.batch) if w.name == "adaptive" else None


def cpu_phases(w, rho, X64, prm, n):
    """Seconds per phase of one oracle run of the global backend on the first
    n tokens, calling the oracle's steps one by one in the order its
    compress_global takes them (features, Lanczos, Ritz pairs, SimHash,
    clusters and adjustment, macro-token means)."""
    import numpy as np
    import oracle as O
    cfg = oracle_config(w, rho)
    Xc = X64[:n - w.preserve_last]
    M = O.target_count(Xc.shape[0], rho)
    bits = cfg.bits if cfg.bits > 0 else O.auto_bits(Xc.shape[0], rho)
    t, out = time.perf_counter(), {}

    def lap(name):
        nonlocal t
        now = time.perf_counter()
        out[name] = now - t
        t = now
    phi = O.rff_features(Xc, prm.w_f64(), prm.b).astype(np.float32).astype(np.float64)
    lap("features")
    a, b_, Q, k = O.lanczos(phi, prm.q1[:Xc.shape[0]], w.r, cfg.lanczos_tol)
    lap("lanczos")
    _, _, U = O.ritz_pairs(a, b_, Q)
    lap("ritz")
    codes = O.simhash(U.astype(np.float32), prm.R[:bits, :k])
    lap("simhash")
    groups = O.adjust_groups(O.bucket(codes), M)
    order = O.order_groups(groups, O.POS_MAX)
    lap("segment")
    O.aggregate_groups(Xc, [groups[i] for i in order], True)
    lap("aggregate")
    return out


def cpu_baseline(w, rho, X64, prm, n, pidx, budget_s=10.0):
    """The oracle as it stands, on the first n tokens of one prompt, repeated
    until about budget_s seconds of CPU work have been timed; then the same
    on one core (a child process with single-threaded BLAS) and, for the
    global backend, the oracle's time per phase."""
    tot, reps = 0.0, 0
    while reps == 0 or tot < budget_s:
        tot += cpu_oracle_step(w, rho, X64, prm, n)
        reps += 1
    kind = "compress_" + w.backend
    res = {"value": n * reps / tot, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
           "sample": f"oracle {kind} (numpy float64, BLAS threads = all cores) on the first "
                     f"{n} tokens of prompt {pidx} of the {w.name} workload, D={w.D} r={w.r} "
                     f"b={w.bits or 'auto'} rho={rho:g}; {reps} run(s), {tot:.1f} s"}
    if not windowed(w):
        res["phases_s"] = {k: round(v, 4) for k, v in cpu_phases(w, rho, X64, prm, n).items()}
    one = single_core_baseline(w, rho, n)
    if one is not None:
        res["single_core"] = one
    return res


def single_core_baseline(w, rho, n, budget_s=8.0):
    """The same oracle sample timed in a child process whose BLAS and OpenMP
    pools have one thread (the variables must be set before numpy loads)."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1",
               MKL_NUM_THREADS="1")
    code = ("import json, bench\n"
            f"print(json.dumps(bench.single_core_child({w.name!r}, {rho!r}, {n}, {budget_s})))")
    try:
        r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env,
                           capture_output=True, text=True, timeout=600)
        return json.loads(r.stdout.strip().splitlines()[-1])
    except Exception:
        return None


def single_core_child(name, rho, n, budget_s):
    w = workload(name)
    p, _ = sample_prompt(w)
    import workloads as WL
    prm = WL.params_for(w)
    X64 = p.x_f64()
    tot, reps = 0.0, 0
    while reps == 0 or tot < budget_s:
        tot += cpu_oracle_step(w, rho, X64, prm, n)
        reps += 1
    return {"value": n * reps / tot, "unit": UNIT, "cores": 1, "runs": reps,
            "seconds": round(tot, 2)}


def run_reference(args, rank, world):
    import workloads as WL
    w = workload(args.workload)
    rho = args.rho or w.rho
    if rank != 0:
        return
    p, pidx = sample_prompt(w)
    prm = WL.params_for(w)
    X64 = p.x_f64()
    n = args.ref_sample
    for _ in range(args.warmup):
        cpu_oracle_step(w, rho, X64, prm, min(n, 512))
    ts = [cpu_oracle_step(w, rho, X64, prm, n) for _ in range(args.steps)]
    tot = sum(ts)
    value = n * args.steps / tot
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": config_dict(w, rho, {"sample_tokens": n}),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(),
                             "kind": "oracle",
                             "sample": f"oracle on the first {n} tokens of prompt {pidx} "
                                       f"per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def device_inputs(w, rank, dev):
    """Embeddings on the device: one prompt, or the adaptive batch of
    w.batch prompts gathered on the device from one bf16 vocabulary table
    (the same rows and ids as workloads.make_prompt).  Returns (X, ids) with
    ids the B x N token ids (numpy int32)."""
    import numpy as np
    import torch
    import workloads as WL
    if w.batch == 1:
        p = WL.make_prompt(w, index=rank)
        X = torch.from_numpy(p.X.view(np.int16)).view(torch.bfloat16).to(dev)
        return X, p.ids.astype(np.int32).reshape(1, w.N)
    ids = [WL.prompt_ids(w, index=i, dup_frac=prompt_dup(w, i)) for i in range(w.batch)]
    uniq, inv = np.unique(np.concatenate(ids), return_inverse=True)
    rows = WL.vocab_rows(WL.DATA_SEED, uniq, w.d).astype(np.float32)
    if w.coherent_frac > 0:
        # coherent windows mix a topic direction into the float32 vocabulary
        # rows on the device, then round to bf16 (the generator's recipe)
        tab = torch.from_numpy(rows).to(dev)
        idx = torch.from_numpy(inv.astype(np.int64)).to(dev)
        X = torch.empty((w.batch, w.N, w.d), dtype=torch.bfloat16, device=dev)
        a = w.coherent_mix
        for i in range(w.batch):
            Xi = tab.index_select(0, idx[i * w.N:(i + 1) * w.N])
            for r0, r1, t in WL.coherent_windows(w, index=i):
                tv = torch.from_numpy(t.astype(np.float32)).to(dev)
                Xi[r0:r1] = a * tv[None, :] + math.sqrt(1.0 - a * a) * Xi[r0:r1]
            X[i] = Xi.to(torch.bfloat16)
        del tab
        return X, np.stack(ids).astype(np.int32)
    table = WL.f32_to_bf16_bits(rows)
    tab = torch.from_numpy(table.view(np.int16)).to(dev)
    idx = torch.from_numpy(inv.astype(np.int64)).to(dev)
    X = tab.index_select(0, idx).view(torch.bfloat16).view(w.batch, w.N, w.d)
    del tab
    return X, np.stack(ids).astype(np.int32)


def vocab_table(X, ids, V, dev):
    """The model's input embedding table as it would sit in HBM: V x d bf16,
    the rows of the prompt's ids taken from X (every other row zero, never
    read), so that table[ids] is X."""
    import numpy as np
    import torch
    d = X.shape[-1]
    uniq, first = np.unique(ids.reshape(-1), return_index=True)
    table = torch.zeros((V, d), dtype=X.dtype, device=dev)
    src = X.reshape(-1, d).index_select(0, torch.from_numpy(first.astype(np.int64)).to(dev))
    table.index_copy_(0, torch.from_numpy(uniq.astype(np.int64)).to(dev), src)
    return table


def make_config(sls, w, rho, normalize=False, phi="f32"):
    phi_code = sls.SLS_BF16 if phi == "bf16" else sls.SLS_F32
    backend = {"adaptive": sls.BACKEND_ADAPTIVE, "local": sls.BACKEND_LOCAL}.get(
        w.backend, sls.BACKEND_GLOBAL)
    return sls.Config.make(backend=backend, rho=rho, D=w.D, r=w.r, bits=w.bits,
                           window=w.window if windowed(w) else 2048,
                           preserve_first=w.preserve_first, preserve_last=w.preserve_last,
                           normalize=int(normalize), phi_dtype=phi_code)


class Run:
    """One workload resident on the device: inputs, parameters, outputs and
    the compress workspace, ready for timed sls_compress calls."""

    def __init__(self, sls, w, rho, rank, dev, normalize=False, phi="f32"):
        import numpy as np
        import torch
        import workloads as WL
        self.sls, self.w, self.rho, self.dev, self.phi = sls, w, rho, dev, phi
        self.X, self.ids = device_inputs(w, rank, dev)
        self.prm = WL.params_for(w)
        self.Wt = torch.from_numpy(self.prm.W.view(np.int16)).view(torch.bfloat16).to(dev)
        self.bt = torch.from_numpy(self.prm.b).to(dev)
        self.Rt = torch.from_numpy(self.prm.R).to(dev)
        self.qt = torch.from_numpy(self.prm.q1).to(dev)
        self.cfg = make_config(sls, w, rho, normalize, phi)
        B, N, d = w.batch, w.N, w.d
        self.M = sls.output_count(self.cfg, N)
        self.ws = sls.Workspace(self.cfg, B, N, d, dev)
        self.out = (torch.empty((B, self.M, d), dtype=torch.float32, device=dev),
                    torch.empty((B, self.M), dtype=torch.int32, device=dev),
                    torch.empty((B, N), dtype=torch.int32, device=dev))
        self.Xin = self.X if w.batch > 1 else self.X.view(1, N, d)

    def step(self, X=None, out=None):
        return self.sls.compress(self.Xin if X is None else X, self.cfg, self.Wt, self.bt,
                                 self.Rt, self.qt, workspace=self.ws,
                                 out=self.out if out is None else out)

    def timed(self, steps, warmup, world):
        """warmup untimed calls, then `steps` calls between CUDA events (max
        over ranks), per-phase events, the launch count and the clocks
        sampled meanwhile."""
        import torch
        import torch.distributed as dist
        sls, w = self.sls, self.w
        for _ in range(warmup):
            res = self.step()
        torch.cuda.synchronize()
        if sls.workspace_status(self.ws) != 0:
            raise RuntimeError("device wait timed out during warm-up")
        B = w.batch
        if windowed(w):
            lens = window_lengths(w)
            route = res[4].cpu().numpy()[:B * len(lens)].reshape(B, len(lens))
            self.lz_tokens = int(sum(int(route[i, k]) * lens[k]
                                     for i in range(B) for k in range(len(lens))))
            self.n_spec = int(route.sum())
        else:
            self.lz_tokens = w.N - w.preserve_first - w.preserve_last
            self.n_spec = 1
        nph = len(sls.PHASES)
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2 * nph)]
              for _ in range(steps)]
        for evs in ev:  # events are created lazily: record each once before use
            for e in evs:
                e.record()
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        bus = str(self.dev.index)
        try:
            u = str(torch.cuda.get_device_properties(self.dev).uuid)
            bus = u if u.startswith("GPU-") else "GPU-" + u
        except Exception:
            pass
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        clocks = Clocks(bus)
        time.sleep(0.3)
        launches0 = sls.launch_count()
        start.record()
        for k in range(steps):
            sls.set_phase_events(ev[k])
            self.step()
        end.record()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        launches = sls.launch_count() - launches0
        clk = clocks.stop()
        sls.set_phase_events(None)
        if sls.workspace_status(self.ws) != 0:
            raise RuntimeError("device wait timed out during the timed region")
        ms = start.elapsed_time(end) / steps
        phases = {name: statistics.mean(ev[k][2 * i].elapsed_time(ev[k][2 * i + 1])
                                        for k in range(steps))
                  for i, name in enumerate(sls.PHASES)}
        ms_max = max_over_ranks([ms], world, self.dev)[0]
        return {"ms": ms_max, "phases": phases, "launches": launches, "clocks": clk,
                "value": world * B * w.N / (ms_max / 1e3)}

    def roofline(self, lanczos_ms):
        """Roofline of the dominant kernel, the persistent Lanczos kernel, over
        the Lanczos phase's CUDA-event time: the two-sweep algorithmic count
        (two sweeps over Phi per step plus the basis traffic) and the count
        of what one fused pass per step must move (one sweep over Phi per
        step plus the basis traffic)."""
        w = self.w
        esz = 2 if self.phi == "bf16" else 4
        alg = lanczos_algorithmic_bytes(self.lz_tokens, w.D, w.r, esz)
        one = lanczos_one_pass_bytes(self.lz_tokens, w.D, w.r, esz)
        lz_s = lanczos_ms / 1e3
        peak, src = peaks()
        achieved = alg / lz_s / 1e9 if lz_s > 0 else 0.0
        ach1 = one / lz_s / 1e9 if lz_s > 0 else 0.0
        roof = {"bound": "hbm", "kernel": "lanczos_kernel", "achieved": achieved, "peak": peak,
                "unit": "GB/s", "frac": achieved / peak, "peak_source": src,
                "algorithmic_bytes": alg, "one_pass_bytes": one,
                "achieved_one_pass": ach1, "frac_one_pass": ach1 / peak, "traffic": None}
        tr = os.path.join(ROOT, "profiles", "lanczos_traffic.json")
        if os.path.exists(tr):
            try:
                with open(tr) as f:
                    t = json.load(f)
                if (t.get("workload") == w.name and t.get("kernel_rev") == LANCZOS_KERNEL_REV
                        and self.phi == "f32" and abs(float(t.get("rho", w.rho)) - self.rho) < 1e-9):
                    roof["traffic"] = t["dram_bytes_per_launch"]
                    if lz_s > 0:
                        roof["traffic_achieved"] = t["dram_bytes_per_launch"] / lz_s / 1e9
                        roof["traffic_frac"] = roof["traffic_achieved"] / peak
            except Exception:
                pass
        return roof


def e2e_measure(run, args, world):
    """The same metric end to end through the public API with host buffers:
    every step copies its embeddings in from pinned host memory and its
    outputs back out (serial and double-buffered patterns), and the path
    from token ids with the embedding table resident on the device."""
    import torch
    sls, w, dev, cfg = run.sls, run.w, run.dev, run.cfg
    Xin, out = run.Xin, run.out
    Xt, pos, t2m = out
    B, N, d = w.batch, w.N, w.d
    Xh = Xin.cpu().pin_memory()

    def host_outs():
        return (torch.empty(Xt.shape, dtype=Xt.dtype).pin_memory(),
                torch.empty(pos.shape, dtype=pos.dtype).pin_memory(),
                torch.empty(t2m.shape, dtype=t2m.dtype).pin_memory())

    def timed(fn, steps):
        # warm-up: the first copies through freshly pinned buffers of a GB or
        # more run several times slower than later ones
        fn(3)
        torch.cuda.synchronize()
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record()
        fn(steps)
        e2.record()
        torch.cuda.synchronize()
        return s2.elapsed_time(e2) / steps

    # serial: copy in, compress, copy out, one after the other
    Xd = torch.empty_like(Xin)
    ho = host_outs()

    def serial(n):
        for _ in range(n):
            Xd.copy_(Xh, non_blocking=True)
            run.step(Xd, out)
            for h, o in zip(ho, out):
                h.copy_(o, non_blocking=True)

    ms_serial = timed(serial, args.e2e_steps)
    # pipelined (the serving pattern): two device buffers; a copy stream
    # brings step k+1's inputs in and takes step k's outputs out while step k
    # compresses on the compute stream
    comp = torch.cuda.current_stream(dev)
    cps = torch.cuda.Stream(device=dev)
    outs = [out, (torch.empty_like(Xt), torch.empty_like(pos), torch.empty_like(t2m))]
    hos = [ho, host_outs()]

    def pipeline(Ih, call):
        Ids = [torch.empty(Ih.shape, dtype=Ih.dtype, device=dev) for _ in range(2)]
        h2d = [torch.cuda.Event() for _ in range(2)]
        done = [torch.cuda.Event() for _ in range(2)]
        d2h = [torch.cuda.Event() for _ in range(2)]

        def go(n):
            cps.wait_stream(comp)
            with torch.cuda.stream(cps):
                Ids[0].copy_(Ih, non_blocking=True)
                h2d[0].record(cps)
            for k in range(n):
                b = k % 2
                if k + 1 < n:
                    nb = (k + 1) % 2
                    with torch.cuda.stream(cps):
                        if k >= 1:
                            cps.wait_event(done[nb])
                        Ids[nb].copy_(Ih, non_blocking=True)
                        h2d[nb].record(cps)
                comp.wait_event(h2d[b])
                if k >= 2:
                    comp.wait_event(d2h[b])
                call(Ids[b], outs[b])
                done[b].record(comp)
                with torch.cuda.stream(cps):
                    cps.wait_event(done[b])
                    for h, o in zip(hos[b], outs[b]):
                        h.copy_(o, non_blocking=True)
                    d2h[b].record(cps)
            comp.wait_stream(cps)
        return go

    ms_pipe = timed(pipeline(Xh, lambda x, o: run.step(x, o)), args.e2e_steps)
    # from token ids: the model's embedding table stays in HBM and only the
    # ids come in; the lookup X = E[ids] runs inside the call (not for the
    # coherent-window workload, whose embeddings are no table rows)
    adaptive = w.batch > 1
    ms_ids = None
    if w.coherent_frac <= 0:
        table = vocab_table(run.X, run.ids, w.V, dev)
        Ih = torch.from_numpy(run.ids if adaptive else run.ids.reshape(N)).pin_memory()
        tws = sls.TokensWorkspace(cfg, table.dtype, B, N, d, dev)
        ms_ids = timed(pipeline(Ih, lambda i, o: sls.compress_tokens(i, table, cfg, run.Wt,
                                                                       run.bt, run.Rt, run.qt,
                                                                       workspace=tws, out=o)),
                       args.e2e_steps)
        del table, tws
    m2 = max_over_ranks([ms_pipe, ms_serial, ms_ids or 0.0], world, dev)
    d2h_bytes = Xt.numel() * 4 + pos.numel() * 4 + t2m.numel() * 4
    pipe_v = world * B * N / (m2[0] / 1e3)
    serial_v = world * B * N / (m2[1] / 1e3)
    # both patterns go through the public API; the faster one is reported
    # (with copies of several GB per step the double-buffered pattern can lose
    # to the serial one)
    pipelined_wins = pipe_v >= serial_v
    return {"value": max(pipe_v, serial_v), "unit": UNIT,
            "h2d_bytes_per_step": Xin.numel() * 2,
            "d2h_bytes_per_step": d2h_bytes,
            "mode": ("pipelined: the copies of step k+1 in and step k out overlap the "
                     "compression of step k on a second stream (double-buffered)")
                    if pipelined_wins else
                    ("serial: copy in, compress, copy out, one after the other (faster "
                     "here than the double-buffered pattern)"),
            "pipelined_value": pipe_v,
            "serial_value": serial_v,
            "from_token_ids": None if ms_ids is None else {
                "value": world * B * N / (m2[2] / 1e3), "unit": UNIT,
                "h2d_bytes_per_step": int(B * N) * 4,
                "d2h_bytes_per_step": d2h_bytes,
                "mode": "double-buffered as above; token ids in, the V x d bf16 embedding "
                        "table resident on the device, lookup inside sls_compress_tokens"}}


def full_config_oracle(run, rho):
    """The oracle's whole pass on the full prompt of a single-prompt
    workload, timed once with all cores and once on one core (a child
    process with single-threaded BLAS), and the end-to-end agreement of the
    GPU pass with it (fraction of identical SimHash codes, adjusted Rand index
    of the token maps; reported, not pinned)."""
    import numpy as np
    import workloads as WL
    from tests.gpu_util import adjusted_rand_index
    import oracle as O
    w, sls = run.w, run.sls
    p = WL.make_prompt(w)
    X64 = p.x_f64()
    cfg = oracle_config(w, rho)
    t = time.perf_counter()
    res = O.compress_global(X64, run.prm.w_f64(), run.prm.b, run.prm.R, run.prm.q1, cfg)
    secs = time.perf_counter() - t
    full = {"value": w.N / secs, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "seconds": round(secs, 2),
            "sample": f"oracle compress_global (numpy float64, all cores) on the whole "
                      f"{w.name} prompt, N={w.N} d={w.d} D={w.D} r={w.r} b={w.bits} "
                      f"rho={rho:g}: the same config as the GPU line"}
    one = single_core_baseline(w, rho, w.N, budget_s=0.0)
    if one is not None:
        full["single_core"] = one
    # GPU codes from the kernels sls_compress runs, its token map from the
    # last timed call
    Nc = w.N - w.preserve_first - w.preserve_last
    Xc = run.X[w.preserve_first:w.preserve_first + Nc]
    phi = sls.feature_map(Xc, run.Wt, run.bt)
    _, U, r_eff, _, _ = sls.lanczos_topr(phi, run.qt[:Nc], w.r)
    codes_g = sls.simhash(U, run.Rt, res.info["bits"], k_dev=r_eff).cpu().numpy().view(np.uint32)
    del phi, U
    run.step()
    t2m = run.out[2][0].cpu().numpy()
    agree = {"workload": w.name,
             "codes_identical": float(np.mean(codes_g == res.info["codes"])),
             "ari_tok2macro": adjusted_rand_index(t2m, res.tok2macro),
             "clusters_gpu": int(np.unique(codes_g).size),
             "clusters_oracle": int(res.info["n_clusters"]),
             "note": "reported, not pinned: float32 Phi and double-float Lanczos on the GPU "
                     "against float64 in the oracle flip SimHash bits whose dot is near zero"}
    return full, agree


def sweep_entry(sls, name, rho, rank, dev, world, steps, warmup):
    """One more workload timed in the same process (20 steps by default):
    tokens/s, ms per step, the Lanczos roofline and the clocks."""
    import torch
    w = workload(name)
    run = Run(sls, w, rho, rank, dev)
    t = run.timed(steps, warmup, world)
    roof = run.roofline(t["phases"]["lanczos"])
    ent = {"workload": name, "N": w.N, "d": w.d, "D": w.D, "r": w.r, "rho": rho,
           "batch": w.batch, "tokens_per_s": t["value"], "ms_per_step": t["ms"],
           "lanczos_ms": t["phases"]["lanczos"], "lanczos_frac": roof["frac"],
           "lanczos_frac_one_pass": roof["frac_one_pass"],
           "lanczos_gbs_one_pass": roof["achieved_one_pass"],
           "phases_ms": t["phases"], "clocks": t["clocks"], "steps": steps,
           "spectral_tokens": run.lz_tokens}
    if windowed(w):
        ent["spectral_windows"] = run.n_spec
    del run
    torch.cuda.empty_cache()
    return ent


def run_native(args, rank, world):
    import torch

    import paper_2607_19368_gb300 as sls

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    rho = args.rho or w.rho
    run = Run(sls, w, rho, rank, dev, args.normalize, args.phi)
    t = run.timed(args.steps, args.warmup, world)
    roof = run.roofline(t["phases"]["lanczos"])
    e2e = None if args.no_e2e else e2e_measure(run, args, world)
    cpu, agree, sweep = None, None, None
    if rank == 0 and world == 1:
        if not args.no_cpu_baseline:
            p, pidx = sample_prompt(w)
            cpu = cpu_baseline(w, rho, p.x_f64(), run.prm, args.cpu_sample, pidx)
            if not windowed(w) and not args.normalize and args.phi == "f32":
                cpu["full_config"], agree = full_config_oracle(run, rho)
    B, N = w.batch, w.N
    n_spec, lz_tokens = run.n_spec, run.lz_tokens
    del run
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and not args.no_sweep and args.workload == "qwen7b" \
            and not args.normalize and args.phi == "f32":
        sweep = [sweep_entry(sls, nm, r_ or workload(nm).rho, rank, dev, world,
                             args.sweep_steps, 3)
                 for nm, r_ in (("mistral7b", None), ("qwen14b", None), ("adaptive", 16.0),
                                ("adaptive_mixed", 8.0))]
    if rank != 0:
        return
    extra = {"parallelism": f"replicas x{world}",
             "inputs": "bf16 embeddings and Omega; float32 Phi; double-float Lanczos vectors"}
    if windowed(w):
        extra.update({"spectral_windows": n_spec, "spectral_tokens": lz_tokens})
    if args.normalize:
        extra["operator"] = "row-normalised (Sec. 3.2 variant, symmetric form)"
    if args.phi == "bf16":
        extra["inputs"] = ("bf16 embeddings and Omega; Phi stored as bf16 (opt-in); "
                           "double-float Lanczos vectors")
    line = {"metric": METRIC, "value": t["value"], "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t["ms"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic",
            "config": config_dict(w, rho, extra),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": t["launches"],
            "clocks": t["clocks"], "phases_ms": t["phases"],
            "lanczos_gbs_algorithmic": roof["achieved"]}
    if agree is not None:
        line["agreement"] = agree
    if sweep is not None:
        line["sweep"] = sweep
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    import torch
    import torch.distributed as dist
    if world > 1:
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist.init_process_group("nccl")
    try:
        run_native(args, rank, world)
    finally:
        if world > 1:
            dist.destroy_process_group()


if __name__ == "__main__":
    main()

"""Benchmark of the Spectral-LSH compression pass on GB300.

One step = one sls_compress call (features, Lanczos, Ritz vectors, SimHash,
clusters/adjust/order, macro-token aggregation) over one synthetic prompt of
the Qwen2.5-7B-shaped workload: N = 32768 tokens, d = 3584 bf16 embeddings,
D = 2048 RFF features, r = 64 Lanczos steps, b = 16 SimHash bits, rho = 16,
last 12 tokens preserved, global backend.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

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
    ap.add_argument("--workload", default="qwen7b")
    ap.add_argument("--cpu-sample", type=int, default=4096,
                    help="tokens of the prompt the CPU oracle compresses per baseline step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--ref-sample", type=int, default=1024,
                    help="tokens the oracle compresses per step of --impl reference")
    return ap.parse_args()


def workload(name):
    import workloads as WL
    return WL.WORKLOADS[name]


def config_dict(w, extra=None):
    d = {"workload": f"{w.name}-shaped prompt: N={w.N} d={w.d} bf16, D={w.D} r={w.r} "
                     f"b={w.bits} rho={int(w.rho)} preserve_last={w.preserve_last}, "
                     f"global backend",
         "N": w.N, "d": w.d, "D": w.D, "r": w.r, "bits": w.bits, "rho": w.rho,
         "l2": "inputs larger than L2 (X 235 MB and Phi 268 MB per step), no flush"}
    if extra:
        d.update(extra)
    return d


# Revision of the persistent Lanczos kernel whose DRAM counters are recorded in
# profiles/lanczos_traffic.json; bumped with every change of the kernel, so a
# stale capture reads as "traffic": null.
LANCZOS_KERNEL_REV = "fused-pass/1"


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


def lanczos_algorithmic_bytes(n_tokens, D, r):
    """Per launch: two float32 sweeps over Phi per step (8 r D bytes per token)
    plus the double-float basis traffic of the two Gram-Schmidt passes
    (16 r (r + 1) bytes per token)."""
    return n_tokens * (8 * r * D + 16 * r * (r + 1))


def cpu_oracle_step(w, X64, prm, n):
    import oracle as O
    cfg = O.CompressConfig(rho=w.rho, D=w.D, r=w.r, bits=w.bits, preserve_last=w.preserve_last)
    t = time.perf_counter()
    O.compress_global(X64[:n], prm.w_f64(), prm.b, prm.R, prm.q1, cfg)
    return time.perf_counter() - t


def cpu_baseline(w, p, prm, n, budget_s=10.0):
    """The oracle as it stands, on the first n tokens of the prompt, repeated
    until about budget_s seconds of CPU work have been timed."""
    X64 = p.x_f64()
    tot, reps = 0.0, 0
    while reps == 0 or tot < budget_s:
        tot += cpu_oracle_step(w, X64, prm, n)
        reps += 1
    return {"value": n * reps / tot, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"oracle compress_global (numpy float64, BLAS threads = all cores) on the "
                      f"first {n} tokens of the {w.name}-shaped prompt, D={w.D} r={w.r} "
                      f"b={w.bits} rho={int(w.rho)}; {reps} run(s), {tot:.1f} s"}


def run_reference(args, rank, world):
    import workloads as WL
    w = workload(args.workload)
    if rank != 0:
        return
    p = WL.make_prompt(w)
    prm = WL.params_for(w)
    X64 = p.x_f64()
    n = args.ref_sample
    for _ in range(args.warmup):
        cpu_oracle_step(w, X64, prm, min(n, 512))
    ts = [cpu_oracle_step(w, X64, prm, n) for _ in range(args.steps)]
    tot = sum(ts)
    value = n * args.steps / tot
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": config_dict(w, {"sample_tokens": n}),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(),
                             "kind": "oracle",
                             "sample": f"oracle compress_global on the first {n} tokens per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_native(args, rank, world):
    import numpy as np
    import torch
    import torch.distributed as dist

    import workloads as WL
    import paper_2607_19368_gb300 as sls

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    p = WL.make_prompt(w, index=rank)
    prm = WL.params_for(w)
    X = torch.from_numpy(p.X.view(np.int16)).view(torch.bfloat16).to(dev)
    Wt = torch.from_numpy(prm.W.view(np.int16)).view(torch.bfloat16).to(dev)
    bt = torch.from_numpy(prm.b).to(dev)
    Rt = torch.from_numpy(prm.R).to(dev)
    qt = torch.from_numpy(prm.q1).to(dev)
    cfg = sls.Config.make(backend=sls.BACKEND_GLOBAL, rho=w.rho, D=w.D, r=w.r, bits=w.bits,
                          preserve_last=w.preserve_last)
    N, d = w.N, w.d
    M = sls.output_count(cfg, N)
    ws = sls.Workspace(cfg, 1, N, d, dev)
    Xt = torch.empty((1, M, d), dtype=torch.float32, device=dev)
    pos = torch.empty((1, M), dtype=torch.int32, device=dev)
    t2m = torch.empty((1, N), dtype=torch.int32, device=dev)
    out = (Xt, pos, t2m)

    def step():
        sls.compress(X, cfg, Wt, bt, Rt, qt, workspace=ws, out=out)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if sls.workspace_status(ws) != 0:
        raise RuntimeError("device wait timed out during warm-up")

    nph = len(sls.PHASES)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2 * nph)]
          for _ in range(args.steps)]
    for evs in ev:  # events are created lazily: record each once before use
        for e in evs:
            e.record()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    bus = str(dev.index)
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
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
    for k in range(args.steps):
        sls.set_phase_events(ev[k])
        step()
    end.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    launches = sls.launch_count() - launches0
    clk = clocks.stop()
    sls.set_phase_events(None)
    if sls.workspace_status(ws) != 0:
        raise RuntimeError("device wait timed out during the timed region")
    ms = start.elapsed_time(end) / args.steps
    phases = {name: statistics.mean(ev[k][2 * i].elapsed_time(ev[k][2 * i + 1])
                                    for k in range(args.steps))
              for i, name in enumerate(sls.PHASES)}
    ms_t = torch.tensor([ms], device=dev)
    if world > 1:
        dist.all_reduce(ms_t, op=dist.ReduceOp.MAX)
    ms_max = float(ms_t.item())
    value = world * N / (ms_max / 1e3)

    # roofline of the dominant kernel (the persistent Lanczos kernel)
    Nc = N - w.preserve_last
    alg = lanczos_algorithmic_bytes(Nc, w.D, w.r)
    lz_s = phases["lanczos"] / 1e3
    peak, src = peaks()
    achieved = alg / lz_s / 1e9
    roof = {"bound": "hbm", "kernel": "lanczos_kernel", "achieved": achieved, "peak": peak,
            "unit": "GB/s", "frac": achieved / peak, "peak_source": src,
            "algorithmic_bytes": alg, "traffic": None}
    tr = os.path.join(ROOT, "profiles", "lanczos_traffic.json")
    if os.path.exists(tr):
        try:
            with open(tr) as f:
                t = json.load(f)
            if t.get("workload") == w.name and t.get("kernel_rev") == LANCZOS_KERNEL_REV:
                roof["traffic"] = t["dram_bytes_per_launch"]
        except Exception:
            pass

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        Xh = X.cpu().pin_memory()
        Xd = torch.empty_like(X)
        Xth = torch.empty(Xt.shape, dtype=Xt.dtype).pin_memory()
        posh = torch.empty(pos.shape, dtype=pos.dtype).pin_memory()
        t2mh = torch.empty(t2m.shape, dtype=t2m.dtype).pin_memory()

        def e2e_step():
            Xd.copy_(Xh, non_blocking=True)
            sls.compress(Xd, cfg, Wt, bt, Rt, qt, workspace=ws, out=out)
            Xth.copy_(Xt, non_blocking=True)
            posh.copy_(pos, non_blocking=True)
            t2mh.copy_(t2m, non_blocking=True)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record()
        for _ in range(args.e2e_steps):
            e2e_step()
        e2.record()
        torch.cuda.synchronize()
        ms2 = s2.elapsed_time(e2) / args.e2e_steps
        m2 = torch.tensor([ms2], device=dev)
        if world > 1:
            dist.all_reduce(m2, op=dist.ReduceOp.MAX)
        e2e = {"value": world * N / (float(m2.item()) / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": X.numel() * 2,
               "d2h_bytes_per_step": Xt.numel() * 4 + pos.numel() * 4 + t2m.numel() * 4}

    if rank != 0:
        return
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        cpu = cpu_baseline(w, p, prm, args.cpu_sample)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic",
            "config": config_dict(w, {"parallelism": f"replicas x{world}",
                                      "inputs": "bf16 embeddings and Omega; float32 Phi; "
                                                "double-float Lanczos vectors"}),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
            "clocks": clk, "phases_ms": phases,
            "lanczos_gbs_algorithmic": achieved}
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

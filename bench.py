#!/usr/bin/env python3
"""Throughput of the MOBO candidate-scoring step on GB300.

One step = one pass of the whole scoring path over one batch of synthetic
input: standardise -> GP fit -> Pareto front (-> boxes) -> posterior ->
acquisition -> top-k, launched by the C-ABI engine on one stream, inputs
resident in HBM. Metric: candidates scored per second (whole job).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the CPU oracle on the same workload

Under torchrun each rank scores its own replica of the workload on its own
GPU (no collective on the data path; weak scaling); rank 0 prints one JSON
line. Between timed steps the L2 is flushed (a 512 MB write outside the
timed events). The `e2e` object times a stream of steps through the
pipelined host-buffer call (boute_engine_step_host_async): every step copies
its inputs in from pinned host memory and its selection out, and one step's
copies overlap the previous step's computation. Monte-Carlo workloads there
use the engine's own base normals, drawn once on the device from a seed
(fixed base samples, as an optimisation loop keeps them), so a step's inputs
are its observations, hyperparameters and candidates.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2602_10729_gb300 import workloads as wl  # noqa: E402

DEFAULT_WORKLOAD = wl.WORKLOADS[1].name
METRIC = "candidates scored/sec (GP posterior + EHVI) at 1 GB300; % of roofline"
UNIT = "candidates/s"
# nominal dense tensor throughput ratio tf32 : bf16 (1.1 : 2.25 PFLOP/s)
TF32_PER_BF16 = 1.1 / 2.25
NUM_SMS = 152


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(
            d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# ---------------------------------------------------------------- inputs
def host_inputs(w: wl.Workload, threads: int = 16):
    X, Y, L, S2, NZ = [], [], [], [], []
    for b in range(w.B):
        x, y = wl.training_set(w, b)
        ls, s2, nz = wl.hyperparameters(w, b)
        X.append(x); Y.append(y); L.append(ls); S2.append(s2); NZ.append(nz)
    Xc = np.stack([wl.candidates(w, b, 0, w.N, threads) for b in range(w.B)])
    eps = (np.stack([wl.base_normals(w, b, 0, w.N, threads) for b in range(w.B)])
           if w.mode == "mc" else None)
    ref = np.tile(wl.ref_point(w), (w.B, 1))
    kc = np.stack([wl.kernel_params(w, b)[1] for b in range(w.B)]) if w.d_tau else None
    return dict(X=np.stack(X), Y=np.stack(Y), ls=np.stack(L), s2=np.stack(S2),
                noise=np.stack(NZ), ref=ref, Xc=Xc, eps=eps, kc=kc)


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.out = os.path.join("/tmp", f"bench_clocks_{os.getpid()}.csv")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(gpu_index)], stdout=open(self.out, "w"),
                stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.out):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.out)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------- roofline
def roofline(w: wl.Workload, stage: str, ms: float, hbm, bf16):
    """Algorithmic work of one launch of the stage's dominant kernel."""
    B, n, d, m, N, S = w.B, w.n, w.d, w.m, w.N, w.S
    if stage == "posterior":
        # triangular L^-1 contraction (n(n+1)/2 MACs) plus the mean column (n MACs)
        flops = B * N * m * (n * (n + 1) + 2 * n)
        peak = bf16 * TF32_PER_BF16
        return dict(bound="tensor", achieved=flops / (ms * 1e-3) / 1e12, peak=peak,
                    unit="TFLOP/s", per_launch=flops, kernel="posterior_kernel")
    if stage == "acquisition" and w.mode == "mc":
        byts = B * N * (m * S * 4 + 2 * m * 4 + 4)
        return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                    per_launch=byts, kernel="mchvi2_kernel" if m == 2 else "mchvi_kernel")
    if stage == "acquisition":
        byts = B * N * (2 * m * 4 + 4)
        return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                    per_launch=byts, kernel="ehvi2d_kernel")
    if stage == "topk":
        byts = B * N * 4
        return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                    per_launch=byts,
                    kernel="warp_topk_kernel" if w.k <= 32 else "segment_topk_kernel")
    if stage == "fit":
        # Cholesky n^3/3 + triangular inverse n^3/3 flops per (problem,
        # objective), fp32 on the CUDA cores of the SMs the fit occupies (one
        # block per problem-objective): 128 FMA lanes x 2 flops x 2.07 GHz each
        flops = B * m * 2 * n ** 3 / 3
        peak = min(B * m, NUM_SMS) * 128 * 2 * 2.07e9 / 1e12
        return dict(bound="alu", achieved=flops / (ms * 1e-3) / 1e12, peak=peak,
                    unit="TFLOP/s", per_launch=flops, kernel="fit32_kernel")
    byts = B * n * m * 8
    return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                per_launch=byts, kernel=stage)


def profiled_traffic(kernel: str, workload: str):
    """dram bytes per launch from the committed ncu summary of this kernel and
    workload, if that summary was taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", f"{kernel}__{workload}.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    mt = re.search(r"traffic_bytes_per_launch\s*[:=]\s*([0-9.eE+]+)", txt)
    ms = re.search(r"source_sha256\s*[:=]\s*([0-9a-f]{16,64})", txt)
    if not mt or not ms:
        return None
    src = re.search(r"source_file\s*[:=]\s*(\S+)", txt)
    if src:
        h = hashlib.sha256(open(os.path.join(ROOT, src.group(1)), "rb").read()).hexdigest()
        if not h.startswith(ms.group(1)):
            return None
    return float(mt.group(1))


# ---------------------------------------------------------------- ranks
def max_over_ranks(x: float, dist=None, device="cpu") -> float:
    """The largest value of x over all ranks (x itself without a process group)."""
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    if dist is not None:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, w: wl.Workload, seconds: float) -> float:
    """Candidates per second over all ranks, each scoring its own replica of
    the workload (B N candidates) in `seconds` (the slowest rank's time)."""
    return world * w.B * w.N / seconds


# ---------------------------------------------------------------- CPU oracle
def oracle_rate(w: wl.Workload, inp, budget_s: float, threads: int = 0, cons=None):
    """The oracle's scoring step (fit, front, posterior, acquisition, top-k)
    on problem 0 over a candidate sample sized to about budget_s seconds
    (cons: the thresholds of a constrained acquisition, or None)."""
    import oracle
    from oracle import pipeline as opl
    threads = threads or oracle.default_threads()
    kern = None if inp["kc"] is None else (w.d_tau, inp["kc"][0])
    tfs = list(w.transforms) or None
    t0 = time.perf_counter()
    fp = opl.fit_problem(inp["X"][0], inp["Y"][0], inp["ls"][0], inp["s2"][0], inp["noise"][0],
                         inp["ref"][0], kernel=kern, transforms=tfs)
    fit_s = time.perf_counter() - t0
    n_try = min(w.N, 2048)
    t0 = time.perf_counter()
    opl.score(fp, inp["Xc"][0, :n_try], w.mode, min(w.k, n_try),
              None if inp["eps"] is None else inp["eps"][0, :n_try], threads, cons=cons)
    per = (time.perf_counter() - t0) / n_try
    sample = int(max(n_try, min(w.N, (budget_s - fit_s) / max(per, 1e-9))))
    t0 = time.perf_counter()
    fp = opl.fit_problem(inp["X"][0], inp["Y"][0], inp["ls"][0], inp["s2"][0], inp["noise"][0],
                         inp["ref"][0], kernel=kern, transforms=tfs)
    opl.score(fp, inp["Xc"][0, :sample], w.mode, min(w.k, sample),
              None if inp["eps"] is None else inp["eps"][0, :sample], threads, cons=cons)
    dt = time.perf_counter() - t0
    return sample / dt, threads, sample, dt


def run_reference(args, w):
    inp = host_inputs(w)
    import oracle
    threads = oracle.default_threads()
    per_step_budget = max(0.5, 150.0 / max(1, args.steps + args.warmup))
    times, samples = [], []
    for i in range(args.warmup + args.steps):
        rate, thr, sample, dt = oracle_rate(w, inp, per_step_budget, threads, args.cons)
        if i >= args.warmup:
            times.append(dt)
            samples.append(sample)
    total = sum(samples)
    value = total / sum(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "n": w.n, "d": w.d, "m": w.m, "N": w.N,
                   "acquisition": w.mode, "S": w.S, "k": w.k, "l2": "n/a (CPU)",
                   **({"constraints": args.constraints} if args.cons else {})},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{samples[0]} of {w.N} candidates of problem 0 per step, "
                                   "full fit + front + posterior + acquisition + top-k"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU arm
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=0, help="0: same as --steps (max 200)")
    ap.add_argument("--constraints", default="",
                    help="comma-separated thresholds on the standardised, minimised objectives "
                         "(constrained acquisition; 'inf' leaves an objective unconstrained)")
    args = ap.parse_args()
    w = wl.by_name(args.workload)
    args.cons = [float(c) for c in args.constraints.split(",")] if args.constraints else None
    if args.cons is not None and len(args.cons) != w.m:
        ap.error(f"--constraints needs {w.m} values")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args, w)
        return

    import torch

    import __graft_entry__
    from paper_2602_10729_gb300 import boute as bt
    __graft_entry__.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    inp = host_inputs(w)
    t = lambda a, dt: None if a is None else torch.as_tensor(a, dtype=dt, device=dev)
    f64, f32 = torch.float64, torch.float32
    dX, dY, dls, ds2, dnz, dref = (t(inp[k], f64) for k in ("X", "Y", "ls", "s2", "noise", "ref"))
    dXc, deps = t(inp["Xc"], f32), t(inp["eps"], f32)
    mode = bt.BOUTE_ACQ_MC_HVI if w.mode == "mc" else bt.BOUTE_ACQ_EHVI2D
    e = bt.Engine(w.B, w.n, w.d, w.m, w.N, mode, w.S, w.k)
    if args.cons is not None:
        bt.boute_engine_set_constraints(e, torch.tensor([args.cons] * w.B, dtype=f64))
    if w.d_tau:  # composite-kernel variant: the paper's kernel and outcome transforms
        bt.boute_engine_set_kernel(e, w.d_tau, inp["kc"])
        bt.boute_engine_set_outcome_transforms(e, list(w.transforms))
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device=dev)
    val = torch.empty((w.B, w.k), dtype=f32, device=dev)
    args_dev = (dX, dY, dls, ds2, dnz, dref, dXc, deps, idx, val)
    # a dedicated stream: the engine replays its step as a CUDA graph there
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(stream)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)

    for _ in range(max(3, args.warmup)):
        bt.boute_engine_step(e, *args_dev)
    torch.cuda.synchronize()

    def barrier():
        if dist:
            dist.barrier()

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    barrier()
    torch.cuda.synchronize()
    l0 = bt.boute_launch_count()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        bt.boute_engine_step_async(e, *args_dev)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    launches = bt.boute_launch_count() - l0
    clk = clocks.stop() if clocks else None
    bt.boute_engine_step(e, *args_dev)  # synchronising step: raises on any recorded device error
    ms = sum(a.elapsed_time(b) for a, b in ev) / args.steps
    ms_max = max_over_ranks(ms, dist, dev)
    value = whole_job_rate(world, w, ms_max * 1e-3)

    # ---- per-stage breakdown: separate steps with stage events (front stage
    # serialised after the fit so that the stages add up) -----------------------
    bt.boute_engine_set_timing(e, True)
    n_stage = min(args.steps, 200)
    stage_ms = {s: 0.0 for s in bt.STAGES}
    for i in range(n_stage + 3):
        flush.zero_()
        bt.boute_engine_step_async(e, *args_dev)
        if i >= 3:
            for s, v in bt.boute_engine_stage_times(e).items():
                stage_ms[s] += v
    stage_ms = {s: v / n_stage for s, v in stage_ms.items()}
    bt.boute_engine_set_timing(e, False)

    # ---- end to end through the public API with host buffers ----------------
    pin = lambda a, dt: None if a is None else torch.as_tensor(a, dtype=dt).pin_memory()
    hX, hY, hls, hs2, hnz, href = (pin(inp[k], f64) for k in ("X", "Y", "ls", "s2", "noise", "ref"))
    hXc = pin(inp["Xc"], f32)
    # Monte-Carlo steps: fixed base normals drawn once on the device from a
    # seed (the engine's own), as an optimisation loop keeps its base samples;
    # a step's host inputs are then the observations, hyperparameters and
    # candidates
    heps = None
    if w.mode == "mc":
        bt.boute_engine_set_normals(e, 1234)
    hidx = torch.empty((w.B, w.k), dtype=torch.int64).pin_memory()
    hval = torch.empty((w.B, w.k), dtype=f32).pin_memory()
    args_host = (hX, hY, hls, hs2, hnz, href, hXc, heps, hidx, hval)
    h2d = sum(a.numel() * a.element_size() for a in args_host[:8] if a is not None)
    d2h = hidx.numel() * 8 + hval.numel() * 4
    # a stream of steps through the pipelined host-input call: each step's
    # copies in overlap the previous step's computation (two device input
    # sets); every step copies its inputs in and its selection out
    bt.boute_engine_step_host(e, *args_host)
    for _ in range(2):  # (captures the graph of each input set)
        bt.boute_engine_step_host_async(e, *args_host)
    bt.boute_engine_sync(e)
    n_e2e = args.e2e_steps or min(args.steps, 200)
    barrier()
    t0 = time.perf_counter()
    for _ in range(n_e2e):
        bt.boute_engine_step_host_async(e, *args_host)
    bt.boute_engine_sync(e)
    e2e_s = (time.perf_counter() - t0) / n_e2e
    e2e_value = whole_job_rate(world, w, max_over_ranks(e2e_s, dist, dev))

    if rank == 0:
        hbm, bf16, bf16s, src = peaks()
        dom = max((s for s in stage_ms if s in ("fit", "posterior", "acquisition", "topk")),
                  key=lambda s: stage_ms[s])
        rf = roofline(w, dom, stage_ms[dom], hbm, bf16)
        roof = {"bound": rf["bound"], "achieved": rf["achieved"], "peak": rf["peak"],
                "unit": rf["unit"], "frac": rf["achieved"] / rf["peak"],
                "traffic": profiled_traffic(rf["kernel"], w.name), "kernel": rf["kernel"],
                "stage": dom, "peak_source": src if rf["bound"] != "alu" else "nominal",
                "algorithmic_per_launch": rf["per_launch"]}
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            rate, thr, sample, dt = oracle_rate(w, inp, 12.0, cons=args.cons)
            cpu = {"value": rate, "unit": UNIT, "cores": thr, "kind": "oracle",
                   "sample": f"{sample} of {w.N} candidates of problem 0 ({dt:.1f} s), full fit "
                             "+ front + posterior + acquisition + top-k"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "n": w.n, "d": w.d, "m": w.m, "N": w.N,
                       "acquisition": w.mode, "S": w.S, "k": w.k,
                       "l2": "flushed between steps (512 MB write)", "parallelism": "replicas",
                       "kernel": "composite" if w.d_tau else "matern52",
                       **({"constraints": args.constraints} if args.cons else {})},
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "call": "boute_engine_step_host_async",
                    "pipelined": True,
                    "normals": "device (boute_engine_set_normals)" if w.mode == "mc" else None},
            "gpu_launches": launches,
            "launches_per_step": bt.boute_engine_launches_per_step(e),
            "stage_ms": stage_ms,
            "wall_s": wall,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    e.free()
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()

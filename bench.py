#!/usr/bin/env python3
"""Throughput of the MOBO candidate-scoring step on GB300.

One step = one pass of the whole scoring path over one batch of synthetic
input: standardise -> GP fit -> Pareto front (-> boxes) -> posterior ->
acquisition -> top-k, launched by the C-ABI engine on one stream, inputs
resident in HBM. Metric: candidates scored per second (whole job). The
default workload is the largest single-GPU one, the 3-objective Monte-Carlo
step (n = 1024, d = 24, N = 4 Mi, S = 256).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the CPU oracle on the same workload

Under torchrun each rank scores its own replica of the workload on its own
GPU (no collective on the data path; weak scaling); rank 0 prints one JSON
line. Between timed steps the L2 is flushed (a 512 MB write outside the
timed events). During the timed steps the engine records live stage events
(its normal concurrent schedule, events on the step's stream only), from
which the scoring pass (posterior + acquisition + top-k) and the dominant
kernel are timed for the `roofline` object.

The `e2e` object times a stream of steps through the pipelined host-buffer
call (boute_engine_step_host_async): every step copies its inputs in from
pinned host memory and its selection out, and one step's copies overlap the
previous step's computation. Its value has the Monte-Carlo base normals
passed in as data with every step (copied from the host); `device_normals`
beside it is the same stream of steps with the engine's own base normals,
drawn once on the device from a seed and held fixed, as an optimisation loop
keeps them.
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

DEFAULT_WORKLOAD = wl.WORKLOADS[3].name
METRIC = "candidates scored/sec (GP posterior + EHVI) at 1 GB300; % of roofline"
UNIT = "candidates/s"
# The posterior contraction's operand type and products per algorithmic
# product: fp16 hi/lo operands, three tcgen05.mma kind::f16 per product
# (hi*hi + hi*lo + lo*hi). Its peak is the measured bf16 peak times the
# nominal dense ratio of the operand type to bf16 (fp16 1 : 1).
CONTRACTION = {"dtype": "f16", "products": 3, "per_bf16": 1.0}
NUM_SMS = 152
FMA_LANES_PER_SM = 128


# The engine's in-sample normals of seed s are drawn under the key s ^ this.
INSAMPLE_KEY = 0x6a09e667f3bcc909


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(
            d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# ---------------------------------------------------------------- inputs
def host_inputs(w: wl.Workload, threads: int = 16, count: int | None = None):
    """The workload's inputs on the host; count: only the first `count`
    candidates (and their normals) of each problem."""
    count = w.N if count is None else min(count, w.N)
    X, Y, L, S2, NZ = [], [], [], [], []
    for b in range(w.B):
        x, y = wl.training_set(w, b)
        ls, s2, nz = wl.hyperparameters(w, b)
        X.append(x); Y.append(y); L.append(ls); S2.append(s2); NZ.append(nz)
    Xc = np.stack([wl.candidates(w, b, 0, count, threads) for b in range(w.B)])
    eps = (np.stack([wl.base_normals(w, b, 0, count, threads) for b in range(w.B)])
           if w.mode in ("mc", "nehvi") else None)
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
def tensor_peak(bf16_tflops: float) -> float:
    """Effective dense peak of the posterior contraction in algorithmic
    TFLOP/s: the operand type's peak (measured bf16 x nominal ratio) divided
    by the tensor-core products issued per algorithmic product."""
    return bf16_tflops * CONTRACTION["per_bf16"] / CONTRACTION["products"]


def contraction_flops(w: wl.Workload) -> float:
    """Algorithmic flops of the posterior: V = K* (L^-1)^T over the lower
    triangle (n(n+1)/2 multiply-adds per candidate and objective) and the mean
    K* alpha (n multiply-adds); the noisy acquisition's joint posterior adds
    the dense H^T k* (n^2) and G^T k* (n S) multiply-adds."""
    per = w.n * (w.n + 1) + 2 * w.n
    if w.mode == "nehvi":
        per += 2 * w.n * w.n + 2 * w.n * w.S
    return float(w.B) * w.N * w.m * per


def pass_bytes(w: wl.Workload) -> float:
    """HBM bytes the scoring pass must move per step: each candidate's
    coordinates (4d), its base normals (4mS, Monte-Carlo) and its score (4)."""
    per = 4 * w.d + (4 * w.m * w.S if w.mode in ("mc", "nehvi") else 0) + 4
    if w.mode == "nehvi":  # the shifts l^T z_s: written by the posterior, read back
        per += 2 * 4 * w.m * w.S
    return float(w.B) * w.N * per


def stage_roofline(w: wl.Workload, stage: str, ms: float, hbm, tens, sm_mhz):
    """Roofline of one stage's kernel from its algorithmic work per launch and
    its measured duration (ms)."""
    B, n, d, m, N, S = w.B, w.n, w.d, w.m, w.N, w.S
    if stage == "posterior":
        flops = contraction_flops(w)
        return dict(bound="tensor", achieved=flops / (ms * 1e-3) / 1e12, peak=tens,
                    unit="TFLOP/s", per_launch=flops, kernel="posterior_kernel")
    if stage == "acquisition":
        per = (m * S * 4 * (2 if w.mode == "nehvi" else 1) if w.mode != "ehvi" else 0) + \
            2 * m * 4 + 4
        byts = float(B) * N * per
        kern = ("ehvi2d_kernel" if w.mode == "ehvi" else "nehvi2_kernel" if w.mode == "nehvi"
                else "mchvi2_kernel" if m == 2 else "mchvi_kernel")
        return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                    per_launch=byts, kernel=kern)
    if stage == "topk":
        byts = float(B) * N * 4
        return dict(bound="hbm", achieved=byts / (ms * 1e-3) / 1e9, peak=hbm, unit="GB/s",
                    per_launch=byts,
                    kernel="warp_topk_kernel" if w.k <= 32 else "segment_topk_kernel")
    # the fit: Cholesky n^3/3 + triangular inverse n^3/3 flops per (problem,
    # objective) in fp32 on the CUDA cores, against the whole GPU's FP32 FMA
    # peak at the clock measured during the run
    flops = float(B) * m * 2 * n ** 3 / 3
    peak = NUM_SMS * FMA_LANES_PER_SM * 2 * (sm_mhz or 2070.0) * 1e6 / 1e12
    return dict(bound="alu", achieved=flops / (ms * 1e-3) / 1e12, peak=peak, unit="TFLOP/s",
                per_launch=flops, kernel="fit32_kernel")


def pass_roofline(w: wl.Workload, ms_pass: float, hbm, tens, tens_tf32):
    """The scoring pass (posterior + acquisition + top-k) against its
    roofline, the slower of the tensor bound (algorithmic contraction flops at
    the contraction's effective peak) and the HBM bound (pass_bytes)."""
    t_tensor = contraction_flops(w) / (tens * 1e12) * 1e3
    t_tf32 = contraction_flops(w) / (tens_tf32 * 1e12) * 1e3
    t_hbm = pass_bytes(w) / (hbm * 1e9) * 1e3
    t_roof = max(t_tensor, t_hbm)
    return {"ms": ms_pass, "bound": "tensor" if t_tensor >= t_hbm else "hbm",
            "t_tensor_ms": t_tensor, "t_hbm_ms": t_hbm, "t_roof_ms": t_roof,
            "frac": t_roof / ms_pass,
            "frac_vs_tf32_over_3": max(t_tf32, t_hbm) / ms_pass,
            "contraction": dict(CONTRACTION)}


def profiled_traffic(kernel: str, workload: str, candidates: int):
    """dram bytes per launch from the committed ncu summary of this kernel and
    workload, if that summary was taken on the current kernel source. A
    summary captured on fewer candidates than the workload's (its
    `captured_candidates`) is scaled to `candidates` in proportion: the
    kernel's DRAM traffic is per candidate (coordinates and normals in,
    results out) plus operands that stay in L2."""
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
    cap = re.search(r"captured_candidates\s*[:=]\s*([0-9]+)", txt)
    scale = candidates / float(cap.group(1)) if cap else 1.0
    return float(mt.group(1)) * scale


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
# candidates of each problem generated for the CPU legs (a bounded sample)
CPU_PREFIX = 1 << 18


def oracle_rate(w: wl.Workload, inp, budget_s: float, threads: int = 0, cons=None,
                sample: int | None = None):
    """The oracle's scoring step (fit, front, posterior, acquisition, top-k)
    on problem 0 over a candidate sample sized to about budget_s seconds (or
    `sample` candidates) of the ones in inp (cons: the thresholds of a
    constrained acquisition, or None)."""
    import oracle
    from oracle import pipeline as opl
    threads = threads or oracle.default_threads()
    if w.mode == "nehvi" and "z" not in inp:  # the engine's in-sample normals (seed 0)
        inp["z"] = oracle.base_normals(INSAMPLE_KEY, 1, w.m * w.S, 1, w.n)[0].reshape(
            w.m, w.S, w.n)
    kern = None if inp["kc"] is None else (w.d_tau, inp["kc"][0])
    tfs = list(w.transforms) or None
    avail = inp["Xc"].shape[1]
    if sample is None:
        t0 = time.perf_counter()
        fp = opl.fit_problem(inp["X"][0], inp["Y"][0], inp["ls"][0], inp["s2"][0],
                             inp["noise"][0], inp["ref"][0], kernel=kern, transforms=tfs)
        fit_s = time.perf_counter() - t0
        n_try = min(avail, 2048)
        t0 = time.perf_counter()
        opl.score(fp, inp["Xc"][0, :n_try], w.mode, min(w.k, n_try),
                  None if inp["eps"] is None else inp["eps"][0, :n_try], threads, cons=cons,
                  z=inp.get("z"))
        per = (time.perf_counter() - t0) / n_try
        sample = int(max(n_try, min(avail, (budget_s - fit_s) / max(per, 1e-9))))
    sample = min(sample, avail)
    t0 = time.perf_counter()
    fp = opl.fit_problem(inp["X"][0], inp["Y"][0], inp["ls"][0], inp["s2"][0], inp["noise"][0],
                         inp["ref"][0], kernel=kern, transforms=tfs)
    opl.score(fp, inp["Xc"][0, :sample], w.mode, min(w.k, sample),
              None if inp["eps"] is None else inp["eps"][0, :sample], threads, cons=cons,
              z=inp.get("z"))
    dt = time.perf_counter() - t0
    return sample / dt, threads, sample, dt


def run_reference(args, w):
    inp = host_inputs(w, count=CPU_PREFIX)
    import oracle
    threads = oracle.default_threads()
    per_step_budget = max(0.5, 150.0 / max(1, args.steps + args.warmup))
    times, samples = [], []
    sample = None  # sized on the first (warm-up) step, then held fixed
    for i in range(max(1, args.warmup) + args.steps):
        rate, thr, sample, dt = oracle_rate(w, inp, per_step_budget, threads, args.cons, sample)
        if i >= max(1, args.warmup):
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
    ap.add_argument("--steps", type=int, default=0,
                    help="timed steps (0: as many as take about 10 s, 20 to 2000)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-serial-stages", action="store_true",
                    help="skip the serialised per-stage breakdown")
    ap.add_argument("--e2e-steps", type=int, default=0, help="0: same as --steps (max 200)")
    ap.add_argument("--noisy", action="store_true",
                    help="score with the noisy acquisition (joint in-sample draws; two "
                         "objectives, n <= 128)")
    ap.add_argument("--candidates", type=int, default=0,
                    help="candidates per problem (0: the workload's N); a smaller N keeps "
                         "profiler captures small")
    ap.add_argument("--constraints", default="",
                    help="comma-separated thresholds on the standardised, minimised objectives "
                         "(constrained acquisition; 'inf' leaves an objective unconstrained)")
    args = ap.parse_args()
    w = wl.by_name(args.workload)
    if args.noisy:
        w = wl.noisy(w)
    if args.candidates:
        w = wl.scaled(w, N=args.candidates)
    args.cons = [float(c) for c in args.constraints.split(",")] if args.constraints else None
    if args.cons is not None and len(args.cons) != w.m:
        ap.error(f"--constraints needs {w.m} values")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        if not args.steps:
            args.steps = 20
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
    mode = {"mc": bt.BOUTE_ACQ_MC_HVI, "nehvi": bt.BOUTE_ACQ_NEHVI}.get(w.mode, bt.BOUTE_ACQ_EHVI2D)
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

    # live stage events in the timed steps (the normal concurrent schedule)
    bt.boute_engine_set_timing(e, bt.TIMING_LIVE)
    for _ in range(max(3, args.warmup)):
        flush.zero_()
        bt.boute_engine_step(e, *args_dev)
    torch.cuda.synchronize()
    if not args.steps:  # about 10 s of timed steps
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        bt.boute_engine_step_async(e, *args_dev)
        a1.record(stream)
        torch.cuda.synchronize()
        args.steps = int(max(20, min(2000, 10.0 / max(a0.elapsed_time(a1) * 1e-3, 1e-6))))
        if dist:  # every rank times the same number of steps
            args.steps = int(max_over_ranks(args.steps, dist, dev))

    def barrier():
        if dist:
            dist.barrier()

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    live = {s_: 0.0 for s_ in bt.STAGES}
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
        # this step's stage events (read before the next step records them;
        # the wait falls between the step's events, outside its device time)
        for s_, v in bt.boute_engine_stage_times(e).items():
            live[s_] += v
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    launches = bt.boute_launch_count() - l0
    clk = clocks.stop() if clocks else None
    bt.boute_engine_set_timing(e, False)
    bt.boute_engine_step(e, *args_dev)  # synchronising step: raises on any recorded device error
    ms = sum(a.elapsed_time(b) for a, b in ev) / args.steps
    ms_max = max_over_ranks(ms, dist, dev)
    value = whole_job_rate(world, w, ms_max * 1e-3)
    live = {s_: v / args.steps for s_, v in live.items()}
    live.pop("front", None)  # (beside the fit in the normal schedule)

    # ---- serialised per-stage breakdown: separate steps with stage events
    # (front stage after the fit, K* built inside the posterior, selection as
    # a launch of its own) so that the stages add up ---------------------------
    stage_ms = None
    if not args.no_serial_stages:
        bt.boute_engine_set_timing(e, bt.TIMING_SERIAL)
        n_stage = min(args.steps, 20)
        stage_ms = {s_: 0.0 for s_ in bt.STAGES}
        for i in range(n_stage + 3):
            flush.zero_()
            bt.boute_engine_step_async(e, *args_dev)
            if i >= 3:
                for s_, v in bt.boute_engine_stage_times(e).items():
                    stage_ms[s_] += v
        stage_ms = {s_: v / n_stage for s_, v in stage_ms.items()}
        bt.boute_engine_set_timing(e, False)
    del deps  # (the resident normals are not needed by the host-input steps)
    args_dev = None

    # ---- end to end through the public API with host buffers ----------------
    pin = lambda a, dt: None if a is None else torch.as_tensor(a, dtype=dt).pin_memory()
    hX, hY, hls, hs2, hnz, href = (pin(inp[k], f64) for k in ("X", "Y", "ls", "s2", "noise", "ref"))
    hXc = pin(inp["Xc"], f32)
    hidx = torch.empty((w.B, w.k), dtype=torch.int64).pin_memory()
    hval = torch.empty((w.B, w.k), dtype=f32).pin_memory()
    n_e2e = args.e2e_steps or min(args.steps, 200)

    def e2e_stream(heps):
        """Candidates per second of a pipelined stream of host-input steps,
        and the bytes each step copies in."""
        args_host = (hX, hY, hls, hs2, hnz, href, hXc, heps, hidx, hval)
        h2d = sum(a.numel() * a.element_size() for a in args_host[:8] if a is not None)
        bt.boute_engine_step_host(e, *args_host)
        for _ in range(2):  # (captures the graph of each input set)
            bt.boute_engine_step_host_async(e, *args_host)
        bt.boute_engine_sync(e)
        barrier()
        t0 = time.perf_counter()
        for _ in range(n_e2e):
            bt.boute_engine_step_host_async(e, *args_host)
        bt.boute_engine_sync(e)
        sec = (time.perf_counter() - t0) / n_e2e
        return whole_job_rate(world, w, max_over_ranks(sec, dist, dev)), h2d

    d2h = hidx.numel() * 8 + hval.numel() * 4
    e2e_value, h2d = e2e_stream(pin(inp["eps"], f32))  # normals passed in every step
    e2e = {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h, "call": "boute_engine_step_host_async",
           "pipelined": True, "steps": n_e2e,
           "normals": "host (copied every step)" if w.mode != "ehvi" else None}
    if w.mode != "ehvi":
        # the engine's own base normals, drawn once on the device from a seed
        bt.boute_engine_set_normals(e, 1234)
        dn_value, dn_h2d = e2e_stream(None)
        e2e["device_normals"] = {"value": dn_value, "unit": UNIT,
                                 "h2d_bytes_per_step": dn_h2d, "d2h_bytes_per_step": d2h,
                                 "normals": "device (boute_engine_set_normals, fixed)"}

    if rank == 0:
        hbm, bf16, bf16s, src = peaks()
        # a kernel inside a long step of back-to-back steps: the sustained peak
        tens = tensor_peak(bf16s)
        tens_tf32 = bf16s * (1.1 / 2.25) / 3
        sm_mhz = (clk or {}).get("sm_mhz")
        dom = max(("fit", "posterior", "acquisition", "topk"), key=lambda s_: live[s_])
        rf = stage_roofline(w, dom, live[dom], hbm, tens, sm_mhz)
        roof = {"bound": rf["bound"], "achieved": rf["achieved"], "peak": rf["peak"],
                "unit": rf["unit"], "frac": rf["achieved"] / rf["peak"],
                "traffic": profiled_traffic(rf["kernel"], w.name, w.B * w.N),
                "kernel": rf["kernel"], "stage": dom, "ms": live[dom],
                "algorithmic_per_launch": rf["per_launch"],
                "peak_source": (f"{src} bf16 sustained x {CONTRACTION['per_bf16']:.4f} "
                                f"({CONTRACTION['dtype']}) / {CONTRACTION['products']} products"
                                if rf["bound"] == "tensor" else
                                f"{src} hbm copy" if rf["bound"] == "hbm" else
                                "nominal: 152 SMs x 128 FMA lanes x 2 x measured SM clock"),
                "pass": pass_roofline(w, live["posterior"] + live["acquisition"] + live["topk"],
                                      hbm, tens, tens_tf32)}
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            cin = host_inputs(w, count=CPU_PREFIX)
            rate, thr, sample, dt = oracle_rate(w, cin, 12.0, cons=args.cons)
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
            "e2e": e2e,
            "gpu_launches": launches,
            "launches_per_step": bt.boute_engine_launches_per_step(e),
            "stage_ms_live": live,
            "stage_ms_serial": stage_ms,
            "wall_s": wall,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    e.free()
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()

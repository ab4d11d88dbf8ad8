"""Seeded synthetic workloads for the MOBO candidate-scoring step.

This module is the ONLY code shared by the CUDA path's tests and the CPU
oracle's tests: it draws training sets, candidate sets and Monte-Carlo base
normals from numpy's PCG64, and holds none of the method's arithmetic (no
standardisation, covariance, posterior, front, hypervolume or selection).

The paper optimises a routing-plus-deployment configuration theta = (tau, c)
(Sec. 5.2, "Overall MOBO workflow") whose objectives come from a simulator and
LLM traces that do not exist here. Its decision vectors are stood in for by
points of the unit cube [0,1]^d, and its two objectives (P95 latency, negated
quality; Sec. 4.3, both minimised) by smooth synthetic functions of x with
additive Gaussian observation noise:

    f1(x) = ||x - c 1||^2 / d      f2(x) = ||x - (1 - c) 1||^2 / d

with c = 0.25, or c_i ~ U[0.1, 0.4] per problem for the batched workload; the
large 2-objective workload adds 0.1 sin(2 pi x_0) to f1, and the 3-objective
workload adds f3(x) = 1 - exp(-||x - 0.5 1||^2 / (0.1 d)). The noise term
"N(0, 1e-4)" is read as variance 1e-4 (standard deviation 0.01).

Composite-kernel variants (`composite(w)`) stand in for the paper's decision
vector theta = (tau, c) more closely: the first d_tau = d // 2 features are
routing features in [0, 1], the rest are deployment features, GPU counts in
{0, .., 4} (the allocations a_{m,n} of Sec. 5.2 S5), and the outcomes are a
positive latency L = exp(f1 + e1) and a quality Q = 1 / (1 + exp(f2 + e2)) in
(0, 1) (to be maximised), with f1, f2 evaluated at x with the counts divided
by 4. The GP then uses the composite kernel with the Log and negated Logit
outcome transforms; its extra hyperparameters (interaction and deployment
outputscales, preference strength beta, preference entries s_{m,n} ~ U[0, 1])
come from `kernel_params`.

Random-access generation: candidates and base normals are drawn in blocks of
CHUNK candidates, block j from SeedSequence([seed, stream, j]), so any slice
of a multi-gigabyte input can be regenerated on its own (the oracle checks
sampled candidates of full-size workloads that way).
"""
from __future__ import annotations

import dataclasses
import math
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

CHUNK = 8192  # candidates per independently seeded block

# stream ids within one seed
_S_TRAIN_X, _S_NOISE, _S_CAND, _S_EPS, _S_SHIFT, _S_PREF, _S_INSAMPLE = 0, 1, 2, 3, 4, 5, 6
MAX_COUNT = 4  # deployment features of composite variants: GPU counts 0 .. MAX_COUNT


@dataclass(frozen=True)
class Workload:
    """One scoring workload: B independent problems, each with n observed
    points in [0,1]^d, m objectives, and N candidates to score."""

    name: str
    B: int
    n: int
    d: int
    m: int
    N: int
    mode: str  # "ehvi" (closed-form 2-objective EHVI) or "mc" (Monte-Carlo HVI)
    S: int  # base normals per candidate per objective (mode "mc"), else 0
    k: int  # top-k per problem
    seeds: tuple  # per-problem seed for training data and candidates
    eps_seed: int  # seed of the base normals (mode "mc")
    sine_term: bool = False  # add 0.1 sin(2 pi x_0) to f1
    shifted: bool = False  # per-problem shift c_i ~ U[0.1, 0.4]
    ref: tuple = field(default=())  # reference point in standardised units
    d_tau: int = 0  # composite kernel: routing features [0, d_tau); 0 = Matern-5/2 kernel
    transforms: tuple = field(default=())  # outcome-transform codes per objective, or ()

    def lengthscale(self) -> float:
        return 0.2 * math.sqrt(self.d)


def _mk(name, B, n, d, m, N, mode, S, k, seeds, eps_seed, **kw):
    return Workload(name, B, n, d, m, N, mode, S, k, tuple(seeds), eps_seed,
                    ref=tuple([1.1] * m), **kw)


#: The five workloads, smallest first. Index 1 is the throughput workload.
WORKLOADS = [
    _mk("tiny-ehvi2d-n32-d6-N4096", 1, 32, 6, 2, 4096, "ehvi", 0, 8, [0], 0),
    _mk("medium-mc2d-n128-d12-N65536-S128", 1, 128, 12, 2, 65536, "mc", 128, 32, [1], 1),
    _mk("large-ehvi2d-n512-d16-N1M", 1, 512, 16, 2, 1 << 20, "ehvi", 0, 64, [2], 0,
        sine_term=True),
    _mk("mc3d-n1024-d24-N4M-S256", 1, 1024, 24, 3, 1 << 22, "mc", 256, 128, [3], 2),
    _mk("batched-ehvi2d-64x-n256-d10-N256K", 64, 256, 10, 2, 1 << 18, "ehvi", 0, 16,
        [100 + i for i in range(64)], 0, shifted=True),
]


def composite(w: Workload) -> Workload:
    """The same shapes with the composite kernel's decision vectors and
    outcomes (routing + deployment features, latency and quality)."""
    codes = (1, 6) + (0,) * (w.m - 2)  # log latency, negated logit quality
    return dataclasses.replace(w, name=w.name + "-composite", d_tau=w.d // 2, transforms=codes)


def noisy(w: Workload) -> Workload:
    """The same shapes scored by the noisy acquisition (joint in-sample draws,
    S per objective; two objectives, n <= 128): mode "nehvi", normals as for
    the Monte-Carlo workloads."""
    if w.m != 2 or w.S < 1:
        raise ValueError("the noisy acquisition needs two objectives and S >= 1")
    return dataclasses.replace(w, name=w.name + "-noisy", mode="nehvi")


def by_name(name: str) -> Workload:
    for w in WORKLOADS:
        if w.name == name:
            return w
        if w.name + "-composite" == name:
            return composite(w)
        if w.name + "-noisy" == name:
            return noisy(w)
    raise KeyError(name)


def scaled(w: Workload, *, N: int | None = None, B: int | None = None,
           n: int | None = None, S: int | None = None) -> Workload:
    """Same recipe at a smaller size (parity cases the oracle finishes fast)."""
    B2 = w.B if B is None else B
    return Workload(w.name + "-scaled", B2, w.n if n is None else n, w.d, w.m,
                    w.N if N is None else N, w.mode, w.S if S is None else S,
                    min(w.k, w.N if N is None else N), w.seeds[:B2], w.eps_seed,
                    w.sine_term, w.shifted, w.ref, w.d_tau, w.transforms)


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key))))


def shift(w: Workload, b: int) -> float:
    if not w.shifted:
        return 0.25
    return float(_rng(w.seeds[b], _S_SHIFT).uniform(0.1, 0.4))


def objectives(w: Workload, b: int, X: np.ndarray) -> np.ndarray:
    """Noise-free synthetic objectives (n x m), all to be minimised."""
    d = X.shape[1]
    c = shift(w, b)
    f1 = ((X - c) ** 2).sum(1) / d
    f2 = ((X - (1.0 - c)) ** 2).sum(1) / d
    if w.sine_term:
        f1 = f1 + 0.1 * np.sin(2.0 * np.pi * X[:, 0])
    cols = [f1, f2]
    if w.m >= 3:
        cols.append(1.0 - np.exp(-((X - 0.5) ** 2).sum(1) / (0.1 * d)))
    if w.m > 3:
        raise ValueError("synthetic objectives defined for m <= 3")
    return np.stack(cols, 1)


def _counts(U: np.ndarray, w: Workload) -> np.ndarray:
    """Composite variants: uniform draws in [0, 1) of the deployment features
    become GPU counts 0 .. MAX_COUNT (in place)."""
    if w.d_tau:
        U[:, w.d_tau:] = np.floor(U[:, w.d_tau:] * (MAX_COUNT + 1))
    return U


def training_set(w: Workload, b: int = 0):
    """Observed points of problem b: X (n x d fp64), raw noisy Y (n x m fp64)."""
    X = _counts(_rng(w.seeds[b], _S_TRAIN_X).random((w.n, w.d)), w)
    noise = _rng(w.seeds[b], _S_NOISE).normal(0.0, 0.01, (w.n, w.m))
    if not w.d_tau:
        return X, objectives(w, b, X) + noise
    Xh = X.copy()
    Xh[:, w.d_tau:] /= MAX_COUNT
    F = objectives(w, b, Xh) + noise
    Y = F.copy()
    Y[:, 0] = np.exp(F[:, 0])  # latency
    Y[:, 1] = 1.0 / (1.0 + np.exp(F[:, 1]))  # quality, to be maximised
    return X, Y


def hyperparameters(w: Workload, b: int = 0):
    """Fixed GP hyperparameters per objective: ARD lengthscales (m x d),
    outputscale (m,), noise variance (m,), in standardised units."""
    ls = np.full((w.m, w.d), w.lengthscale())
    if w.d_tau:
        ls[:, w.d_tau:] *= MAX_COUNT  # the deployment features span 0 .. MAX_COUNT
    return ls, np.ones(w.m), np.full(w.m, 1e-4)


def kernel_params(w: Workload, b: int = 0):
    """Composite variants: (d_tau, kc), kc m x (3 + d - d_tau), per objective
    [deployment outputscale, interaction outputscale (phi), beta, preference
    entries ~ U[0, 1]]; None for the Matern-5/2 workloads."""
    if not w.d_tau:
        return None
    dc = w.d - w.d_tau
    pref = _rng(w.seeds[b], _S_PREF).random((w.m, dc))
    kc = np.concatenate([np.tile([0.5, 0.1, 0.05], (w.m, 1)), pref], 1)
    return w.d_tau, kc


def ref_point(w: Workload) -> np.ndarray:
    return np.asarray(w.ref, dtype=np.float64)


def _blocks(start: int, count: int):
    j0, j1 = start // CHUNK, (start + count - 1) // CHUNK
    for j in range(j0, j1 + 1):
        lo, hi = max(start, j * CHUNK), min(start + count, (j + 1) * CHUNK)
        yield j, lo - j * CHUNK, hi - j * CHUNK, lo - start


def _fill(out, start, count, make, threads):
    if count <= 0:
        return out
    jobs = list(_blocks(start, count))

    def one(job):
        j, a, e, o = job
        out[o:o + (e - a)] = make(j)[a:e]

    if threads > 1 and len(jobs) > 1:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(one, jobs))
    else:
        for job in jobs:
            one(job)
    return out


def candidates(w: Workload, b: int, start: int = 0, count: int | None = None,
               threads: int = 1) -> np.ndarray:
    """Candidates [start, start+count) of problem b: U[0,1]^d drawn in fp64 and
    rounded once to fp32 (count x d float32)."""
    count = w.N - start if count is None else count
    out = np.empty((count, w.d), np.float32)
    return _fill(out, start, count,
                 lambda j: _counts(_rng(w.seeds[b], _S_CAND, j).random((CHUNK, w.d)),
                                   w).astype(np.float32), threads)


def insample_normals(w: Workload, b: int, S: int | None = None) -> np.ndarray:
    """Standard-normal base samples of the in-sample draws of problem b (the
    noisy acquisition), fp32, layout (m, S, n)."""
    S = w.S if S is None else S
    return _rng(w.seeds[b], _S_INSAMPLE, w.eps_seed).standard_normal(
        (w.m, S, w.n)).astype(np.float32)


def base_normals(w: Workload, b: int, start: int = 0, count: int | None = None,
                 threads: int = 1) -> np.ndarray:
    """Standard-normal base samples for candidates [start, start+count) of
    problem b, fp32, layout (count, m, S): for each candidate, m rows of S."""
    count = w.N - start if count is None else count
    out = np.empty((count, w.m, w.S), np.float32)
    return _fill(out, start, count,
                 lambda j: _rng(w.eps_seed, w.seeds[b], _S_EPS, j).standard_normal(
                     (CHUNK, w.m, w.S), dtype=np.float32), threads)

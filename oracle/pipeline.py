"""The scoring step composed from oracle functions (test infrastructure only).

Follows the order of one MOBO iteration (Sec. 5.2, "Overall MOBO workflow"):
standardise the observed outcomes, fit one exact GP per objective
(independent GPs combined as a model list, Sec. 6), take the Pareto front of
the observed outcomes, evaluate the posterior and the acquisition at every
candidate, and select the best k.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import (JOINT_JITTER, ehvi2d, gp_fit, gp_posterior, joint_draws, mc_hvi, nehvi_mc,
               outcome_transform, pareto_front, standardize, topk)


@dataclass
class FittedProblem:
    X: np.ndarray  # n x d observed points
    Ys: np.ndarray  # n x m standardised outcomes
    ls: np.ndarray  # m x d
    s2: np.ndarray  # m
    noise: np.ndarray  # m
    L: list  # per objective, n x n
    alpha: list  # per objective, n
    ref: np.ndarray
    mask: np.ndarray  # front membership (n,)
    front: np.ndarray  # P x m, sorted
    kernel: list | None = None  # per objective (dtau, kc) of the composite kernel, or None


def fit_problem(X, Y, ls, s2, noise, ref, kernel=None, transforms=None) -> FittedProblem:
    """kernel: None (Matern-5/2) or (dtau, kc) with kc m x (3 + d - dtau), one
    row [s2_c, s2_x, beta, pref...] per objective (the composite kernel);
    transforms: None or m outcome-transform codes applied before Standardize."""
    if transforms is not None:
        Y = outcome_transform(Y, transforms)
    Ys = standardize(Y)
    kern = None if kernel is None else [(kernel[0], np.asarray(kernel[1], np.float64)[t])
                                        for t in range(Ys.shape[1])]
    Ls, alphas = [], []
    for t in range(Ys.shape[1]):
        L, a = gp_fit(X, Ys[:, t], ls[t], s2[t], noise[t], None if kern is None else kern[t])
        Ls.append(L)
        alphas.append(a)
    mask, order = pareto_front(Ys, ref)
    return FittedProblem(np.asarray(X, np.float64), Ys, np.asarray(ls, np.float64),
                         np.asarray(s2, np.float64), np.asarray(noise, np.float64), Ls, alphas,
                         np.asarray(ref, np.float64), mask, Ys[order], kern)


def posterior(fp: FittedProblem, Xc, threads: int = 0):
    """mean, var: N x m (fp64)."""
    Xc = np.ascontiguousarray(Xc, np.float32)
    m = fp.Ys.shape[1]
    mean = np.empty((Xc.shape[0], m))
    var = np.empty((Xc.shape[0], m))
    for t in range(m):
        mean[:, t], var[:, t] = gp_posterior(fp.X, fp.ls[t], fp.s2[t], fp.L[t], fp.alpha[t], Xc,
                                             threads, None if fp.kernel is None else fp.kernel[t])
    return mean, var


def acquisition(fp: FittedProblem, mean, var, mode: str, eps=None, threads: int = 0,
                cons=None):
    """cons: per-objective feasibility thresholds (standardised units) or None."""
    if mode == "ehvi":
        return ehvi2d(mean, var, fp.front, fp.ref, threads, cons=cons)
    if mode == "mc":
        return mc_hvi(mean, var, eps, fp.front, fp.ref, threads=threads, cons=cons)
    raise ValueError(mode)


def score(fp: FittedProblem, Xc, mode: str, k: int, eps=None, threads: int = 0, cons=None,
          z=None):
    """mode "nehvi": the noisy acquisition with in-sample normals z (m, S, n);
    mean and var are then the marginal mean and the conditional variance."""
    if mode == "nehvi":
        dr, acq, idx, val = noisy_score(fp, Xc, z, eps, k, threads, cons)
        return dr.mean, dr.cvar, acq, idx, val
    mean, var = posterior(fp, Xc, threads)
    acq = acquisition(fp, mean, var, mode, eps, threads, cons=cons)
    idx, val = topk(acq, k)
    return mean, var, acq, idx, val


@dataclass
class NoisyDraws:
    Yin: np.ndarray  # S x n x m in-sample joint draws
    mean: np.ndarray  # N x m
    cvar: np.ndarray  # N x m, variance left once the in-sample values are drawn
    shift: np.ndarray  # N x m x S


def noisy_draws(fp: FittedProblem, Xc, z, jitter: float = JOINT_JITTER,
                threads: int = 0) -> NoisyDraws:
    """Joint posterior draws of every objective (independent GPs, Sec. 6) at
    the observed points and the candidates. z: (m, S, n) float32 in-sample
    normals."""
    Xc = np.ascontiguousarray(Xc, np.float32)
    m = fp.Ys.shape[1]
    z = np.asarray(z, np.float32)
    S, n = z.shape[1], z.shape[2]
    N = Xc.shape[0]
    Yin = np.empty((S, n, m))
    mean = np.empty((N, m))
    cvar = np.empty((N, m))
    shift = np.empty((N, m, S))
    for t in range(m):
        Yin[:, :, t], mean[:, t], cvar[:, t], shift[:, t, :] = joint_draws(
            fp.X, fp.Ys[:, t], fp.ls[t], fp.s2[t], fp.noise[t], z[t], Xc, jitter, threads,
            None if fp.kernel is None else fp.kernel[t])
    return NoisyDraws(Yin, mean, cvar, shift)


def noisy_acquisition(fp: FittedProblem, dr: NoisyDraws, eps, threads: int = 0, cons=None):
    """Noisy MC hypervolume improvement of every candidate (Sec. 5.2,
    constrained qNEHVI, q = 1): the front of each sample is that of its
    feasible in-sample draws."""
    return nehvi_mc(dr.Yin, dr.mean, dr.cvar, dr.shift, eps, fp.ref, threads, cons=cons)


def noisy_score(fp: FittedProblem, Xc, z, eps, k: int, threads: int = 0, cons=None,
                jitter: float = JOINT_JITTER):
    dr = noisy_draws(fp, Xc, z, jitter, threads)
    acq = noisy_acquisition(fp, dr, eps, threads, cons)
    idx, val = topk(acq, k)
    return dr, acq, idx, val

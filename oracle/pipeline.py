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


# ---- optimising the acquisition over the decision space (Sec. 5.2 step (ii)) -----
# The Monte-Carlo hypervolume improvement with fixed base normals (a sample
# average, so that the acquisition is a deterministic, piecewise smooth
# function of the point x), its gradient through the GP posterior, and
# projected Adam ascent from given starting points. Two objectives, the
# Matern-5/2 kernel, the observed front.
_SQRT5 = 5.0 ** 0.5


def _kstar_grad(X, ls, s2, x):
    """k*_j = s2 (1 + sqrt5 r + 5/3 r^2) exp(-sqrt5 r) at the scaled distance r
    of x to X_j, and its gradient in x: dk*_j/dx = -5/3 s2 (1 + sqrt5 r)
    exp(-sqrt5 r) (x - X_j) / ls^2 (n x d)."""
    diff = (x[None, :] - X) / ls
    r = np.sqrt((diff * diff).sum(1))
    ex = np.exp(-_SQRT5 * r)
    k = s2 * (1.0 + _SQRT5 * r + 5.0 / 3.0 * r * r) * ex
    dk = (-5.0 / 3.0 * s2 * (1.0 + _SQRT5 * r) * ex)[:, None] * diff / ls[None, :]
    return k, dk


def _forward(L, b):
    x = np.empty_like(b)
    for i in range(len(b)):
        x[i] = (b[i] - L[i, :i] @ x[:i]) / L[i, i]
    return x


def _backward(L, b):  # solves L^T x = b
    n = len(b)
    x = np.empty_like(b)
    for i in range(n - 1, -1, -1):
        x[i] = (b[i] - L[i + 1:, i] @ x[i + 1:]) / L[i, i]
    return x


def posterior_grad(fp: FittedProblem, t: int, x):
    """Posterior mean and variance of objective t at x and their gradients:
    mean = k*^T alpha, var = s2 - v^T v with v = L^-1 k*, d var/dx = -2
    (K^-1 k*)^T dk*/dx."""
    k, dk = _kstar_grad(fp.X, fp.ls[t], fp.s2[t], np.asarray(x, np.float64))
    mean = k @ fp.alpha[t]
    dmean = dk.T @ fp.alpha[t]
    v = _forward(fp.L[t], k)
    var = fp.s2[t] - v @ v
    kinv_k = _backward(fp.L[t], v)
    dvar = -2.0 * dk.T @ kinv_k
    return mean, var, dmean, dvar


def _strips(front, ref):
    """The undominated region of a 2-D front (f1 ascending) as strips
    (a_k, b_k, u_k): x in [a_k, b_k), y below u_k."""
    P = len(front)
    a = np.concatenate([[-np.inf], front[:, 0]])
    b = np.concatenate([front[:, 0], [ref[0]]]) if P else np.array([ref[0]])
    u = np.concatenate([[ref[1]], front[:, 1]])
    return a, b, u


def hvi2_grad(front, ref, y):
    """Hypervolume improvement of y over a 2-D front and its gradient in y:
    HVI = sum_k (b_k - max(a_k, y1))+ (u_k - y2)+."""
    a, b, u = _strips(front, ref)
    w = np.maximum(b - np.maximum(a, y[0]), 0.0)
    h = np.maximum(u - y[1], 0.0)
    val = float((w * h).sum())
    inside = (a < y[0]) & (y[0] < b)
    g1 = -float((inside * h).sum())
    g2 = -float((w * (y[1] < u)).sum())
    return val, np.array([g1, g2])


def mc_hvi_value_grad(fp: FittedProblem, x, eps):
    """The sample-average acquisition (1/S) sum_s HVI(mean + sd eps_s) at x,
    eps: (2, S) base normals, and its gradient in x (the chain through the
    posterior mean and standard deviation of both objectives)."""
    x = np.asarray(x, np.float64)
    eps = np.asarray(eps, np.float64)
    S = eps.shape[1]
    mu, sd, dmu, dsd = [], [], [], []
    for t in range(2):
        m_, v_, dm_, dv_ = posterior_grad(fp, t, x)
        s_ = np.sqrt(max(v_, 0.0))
        mu.append(m_)
        sd.append(s_)
        dmu.append(dm_)
        dsd.append(dv_ / (2.0 * s_) if s_ > 0 else np.zeros_like(dv_))
    val, grad = 0.0, np.zeros_like(x)
    for s in range(S):
        y = np.array([mu[0] + sd[0] * eps[0, s], mu[1] + sd[1] * eps[1, s]])
        h, g = hvi2_grad(fp.front, fp.ref, y)
        val += h
        grad += g[0] * (dmu[0] + eps[0, s] * dsd[0]) + g[1] * (dmu[1] + eps[1, s] * dsd[1])
    return val / S, grad / S


def optimize_acq(fp: FittedProblem, X0, eps, lower, upper, steps: int, lr: float):
    """Projected Adam ascent (beta1 0.9, beta2 0.999, eps 1e-8) on
    mc_hvi_value_grad from each row of X0, every iterate clamped to
    [lower, upper]. Returns the final points and their acquisition values."""
    X = np.array(X0, np.float64, copy=True)
    out = np.empty(len(X))
    for p in range(len(X)):
        x = X[p]
        m1 = np.zeros_like(x)
        m2 = np.zeros_like(x)
        for it in range(1, steps + 1):
            _, g = mc_hvi_value_grad(fp, x, eps)
            m1 = 0.9 * m1 + 0.1 * g
            m2 = 0.999 * m2 + 0.001 * g * g
            step = lr * (m1 / (1 - 0.9 ** it)) / (np.sqrt(m2 / (1 - 0.999 ** it)) + 1e-8)
            x = np.clip(x + step, lower, upper)
        X[p] = x
        out[p] = mc_hvi_value_grad(fp, x, eps)[0]
    return X, out

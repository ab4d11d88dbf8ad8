"""Pins of the oracle's noisy acquisition (Sec. 5.2, constrained qNEHVI: the
expectation over the joint posterior of the objectives at the observed points
and at the candidate) against facts that do not come from the oracle:

* the draws equal those of the Cholesky factor of the full joint posterior
  covariance of (f(X), f(x)), built here with numpy from the GP's definition
  and a Bessel-function route to the Matern kernel (the factor is unique);
* the per-sample fronts, feasibility and averaging equal a brute-force
  hypervolume over a coordinate-compressed grid;
* the Monte-Carlo estimate agrees, within its standard error, with one from
  numpy's own multivariate-normal sampler of the same joint distribution;
* with (almost) no observation noise the in-sample draws collapse onto the
  observations and the acquisition becomes the MC-HVI against the observed
  front."""
import math

import numpy as np
import pytest
import scipy.special

import oracle
from oracle import pipeline


def _matern52_bessel(a, b, ls, s2):
    r = float(np.sqrt((((np.asarray(a) - np.asarray(b)) / ls) ** 2).sum()))
    if r == 0:
        return s2
    nu = 2.5
    zz = math.sqrt(2 * nu) * r
    return s2 * 2 ** (1 - nu) / scipy.special.gamma(nu) * zz ** nu * scipy.special.kv(nu, zz)


def _joint_cov(X, x, y, ls, s2, noise):
    """Mean and covariance of (f(X), f(x)) given y = f(X) + noise, from the
    definitions: mu = K_pX (K_XX + noise I)^-1 y, C = K_pp - K_pX (.)^-1 K_Xp."""
    P = np.vstack([X, x[None, :]])
    Kpp = np.array([[_matern52_bessel(a, b, ls, s2) for b in P] for a in P])
    n = len(X)
    KXX = Kpp[:n, :n] + noise * np.eye(n)
    KpX = Kpp[:, :n]
    mu = KpX @ np.linalg.solve(KXX, y)
    C = Kpp - KpX @ np.linalg.solve(KXX, KpX.T)
    return mu, (C + C.T) / 2


def _problem(seed, n=5, d=2, N=3, S=4, noise=2e-2):
    rng = np.random.default_rng(seed)
    X = rng.random((n, d))
    y = rng.standard_normal(n)
    ls = rng.uniform(0.3, 0.9, d)
    z = rng.standard_normal((S, n)).astype(np.float32)
    Xc = rng.random((N, d)).astype(np.float32)
    eps = rng.standard_normal((N, S)).astype(np.float32)
    return X, y, ls, 1.3, noise, z, Xc, eps


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_joint_draws_equal_full_joint_cholesky(seed):
    X, y, ls, s2, noise, z, Xc, eps = _problem(seed)
    n, S = len(X), z.shape[0]
    jit = 1e-6
    Yin, mean, cvar, shift = oracle.joint_draws(X, y, ls, s2, noise, z, Xc, jitter=jit)
    for c in range(len(Xc)):
        mu, C = _joint_cov(X, Xc[c].astype(np.float64), y, ls, s2, noise)
        C[np.arange(n), np.arange(n)] += jit * s2  # the jitter on the in-sample block
        Lj = np.linalg.cholesky(C)
        for s in range(S):
            w = np.concatenate([z[s].astype(np.float64), [float(eps[c, s])]])
            draw = mu + Lj @ w
            np.testing.assert_allclose(Yin[s], draw[:n], rtol=1e-9, atol=1e-11)
            got = mean[c] + shift[c, s] + math.sqrt(max(cvar[c], 0.0)) * float(eps[c, s])
            assert got == pytest.approx(draw[n], rel=1e-9, abs=1e-11)
        # the conditional variance is the last pivot squared
        assert cvar[c] == pytest.approx(Lj[n, n] ** 2, rel=1e-8, abs=1e-13)
        assert mean[c] == pytest.approx(mu[n], rel=1e-10, abs=1e-12)


def _hv_grid(pts, ref):
    """Exact 2-D hypervolume (minimisation) of a point set by summing the
    cells of the grid of all coordinates that some point dominates."""
    pts = [p for p in pts if p[0] < ref[0] and p[1] < ref[1]]
    if not pts:
        return 0.0
    xs = sorted({p[0] for p in pts} | {ref[0]})
    ys = sorted({p[1] for p in pts} | {ref[1]})
    area = 0.0
    for i in range(len(xs) - 1):
        for j in range(len(ys) - 1):
            if any(p[0] <= xs[i] and p[1] <= ys[j] for p in pts):
                area += (xs[i + 1] - xs[i]) * (ys[j + 1] - ys[j])
    return area


def _brute_nehvi(Yin, ys, ref, cons):
    """Yin: (S, n, 2); ys: (N, 2, S) candidate draws."""
    S = Yin.shape[0]
    out = []
    for c in range(ys.shape[0]):
        tot = 0.0
        for s in range(S):
            base = [p for p in Yin[s] if cons is None or (p[0] <= cons[0] and p[1] <= cons[1])]
            y = ys[c, :, s]
            if cons is not None and not (y[0] <= cons[0] and y[1] <= cons[1]):
                continue
            tot += _hv_grid(base + [y], ref) - _hv_grid(base, ref)
        out.append(tot / S)
    return np.array(out)


@pytest.mark.parametrize("cons", [None, (0.3, 0.6)])
def test_nehvi_equals_brute_force_over_samples(cons):
    rng = np.random.default_rng(7)
    S, n, N = 6, 7, 5
    Yin = rng.standard_normal((S, n, 2)) * 0.5
    mean = rng.standard_normal((N, 2)) * 0.5
    cvar = rng.uniform(0.01, 0.2, (N, 2))
    cvar[0, 1] = -1e-9  # a rounding-negative variance counts as zero
    shift = rng.standard_normal((N, 2, S)) * 0.1
    eps = rng.standard_normal((N, 2, S)).astype(np.float32)
    ref = np.array([1.0, 1.2])
    acq = oracle.nehvi_mc(Yin, mean, cvar, shift, eps, ref, cons=cons)
    ys = mean[:, :, None] + shift + np.sqrt(np.maximum(cvar, 0))[:, :, None] * eps
    want = _brute_nehvi(Yin, ys, ref, cons)
    np.testing.assert_allclose(acq, want, rtol=1e-10, atol=1e-13)
    assert (acq >= 0).all()


def test_mc_estimate_agrees_with_independent_joint_sampler():
    """The expectation the oracle estimates is that of the joint posterior:
    compare with numpy's multivariate-normal draws of (f(X), f(x)) for both
    objectives (independent GPs), within 5 standard errors."""
    rng = np.random.default_rng(11)
    n, d, S = 4, 2, 20000
    X = rng.random((n, d))
    Y = rng.standard_normal((n, 2)) * 0.6
    ls = np.array([[0.6, 0.8], [0.7, 0.5]])
    s2, noise = np.array([1.0, 0.8]), np.array([0.05, 0.1])
    x = np.array([0.45, 0.55], np.float32)
    ref = np.array([1.5, 1.5])
    z = rng.standard_normal((2, S, n)).astype(np.float32)
    eps = rng.standard_normal((1, 2, S)).astype(np.float32)
    parts = [oracle.joint_draws(X, Y[:, t], ls[t], s2[t], noise[t], z[t], x[None, :])
             for t in range(2)]
    Yin = np.stack([p[0] for p in parts], -1)
    mean = np.array([[p[1][0] for p in parts]])
    cvar = np.array([[p[2][0] for p in parts]])
    shift = np.stack([p[3] for p in parts], 1)
    acq = oracle.nehvi_mc(Yin, mean, cvar, shift, eps, ref)[0]
    # independent: numpy's sampler on the joint covariance (no jitter needed)
    rng2 = np.random.default_rng(12)
    draws = []
    for t in range(2):
        mu, C = _joint_cov(X, x.astype(np.float64), Y[:, t], ls[t], s2[t], noise[t])
        draws.append(rng2.multivariate_normal(mu, C, size=S, method="eigh"))
    D = np.stack(draws, -1)  # S x (n + 1) x 2
    vals = np.empty(S)
    for s in range(S):
        base = [tuple(p) for p in D[s, :n]]
        y = tuple(D[s, n])
        vals[s] = _hv_fast(base + [y], ref) - _hv_fast(base, ref)
    se = vals.std() / math.sqrt(S)
    assert abs(acq - vals.mean()) < 5 * se + 1e-12, (acq, vals.mean(), se)
    assert acq > 10 * se  # the comparison is not vacuous


def _hv_fast(pts, ref):
    """2-D hypervolume by the staircase sweep (checked against _hv_grid)."""
    pts = sorted(p for p in pts if p[0] < ref[0] and p[1] < ref[1])
    hv, cur = 0.0, ref[1]
    for p in pts:
        if p[1] < cur:
            hv += (ref[0] - p[0]) * (cur - p[1])
            cur = p[1]
    return hv


def test_hv_fast_matches_grid():
    rng = np.random.default_rng(3)
    for _ in range(50):
        pts = [tuple(p) for p in rng.standard_normal((6, 2))]
        assert _hv_fast(pts, (1.0, 1.0)) == pytest.approx(_hv_grid(pts, (1.0, 1.0)), abs=1e-12)


def test_noiseless_limit_is_mc_hvi_against_observed_front():
    """noise -> 0: the in-sample posterior collapses onto the observations,
    the candidate's draw onto its marginal; the acquisition becomes the MC-HVI
    of the observed front (the oracle's pinned mc_hvi)."""
    rng = np.random.default_rng(5)
    n, d, N, S = 12, 3, 40, 16
    X = rng.random((n, d))
    Y = np.stack([((X - 0.3) ** 2).sum(1), ((X - 0.7) ** 2).sum(1)], 1)
    ls = np.full((2, d), 0.4)
    s2, noise = np.ones(2), np.full(2, 1e-9)
    ref = np.array([1.2, 1.2])
    fp = pipeline.fit_problem(X, Y, ls, s2, noise, ref)
    Xc = rng.random((N, d)).astype(np.float32)
    z = rng.standard_normal((2, S, n)).astype(np.float32)
    eps = rng.standard_normal((N, 2, S)).astype(np.float32)
    dr = pipeline.noisy_draws(fp, Xc, z, jitter=1e-13)
    np.testing.assert_allclose(dr.Yin, np.broadcast_to(fp.Ys, dr.Yin.shape), atol=5e-4)
    mean, var = pipeline.posterior(fp, Xc)
    np.testing.assert_allclose(dr.mean, mean, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dr.cvar, var, atol=1e-6)
    assert abs(dr.shift).max() < 5e-3
    got = pipeline.noisy_acquisition(fp, dr, eps)
    want = oracle.mc_hvi(mean, var, eps, fp.front, ref)
    assert abs(got - want).max() < 2e-2 * max(want.max(), 1e-3)
    assert want.max() > 0

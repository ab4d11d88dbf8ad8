"""Pins of the oracle's acquisition gradient and optimiser (Sec. 5.2 step
(ii): the acquisition optimised over the decision space) against facts that
do not come from that code: central differences of the C oracle's posterior
and Monte-Carlo HVI (themselves pinned in test_oracle_pins.py), the C
oracle's HVI, and a dense grid search of the acquisition on a
one-dimensional problem. Finite differences use steps that are exact in fp32
(the C oracle takes fp32 points), and points where some draw crosses a strip
edge inside the step (a kink of the sample average) are skipped."""
import numpy as np
import pytest

import oracle
from oracle import pipeline as opl

H = 2.0 ** -14


def _problem(seed, n=12, d=3):
    rng = np.random.default_rng(seed)
    X = rng.random((n, d))
    Y = np.stack([((X - 0.3) ** 2).sum(1), ((X - 0.7) ** 2).sum(1)], 1) + 0.01 * rng.standard_normal((n, 2))
    ls = np.full((2, d), 0.5)
    fp = opl.fit_problem(X, Y, ls, np.ones(2), np.full(2, 1e-3), np.array([1.2, 1.2]))
    eps = rng.standard_normal((2, 32)).astype(np.float32).astype(np.float64)
    return fp, eps, rng


def _acq_c(fp, eps, x):
    """The acquisition from the C oracle: posterior at the fp32 point, MC-HVI
    with the (fp32) normals shared by the point."""
    mean, var = opl.posterior(fp, np.asarray(x, np.float32)[None])
    e = eps.astype(np.float32)[None]  # (1, 2, S)
    return oracle.mc_hvi(mean, var, e, fp.front, fp.ref)[0]


def _fd(f, x, h):
    g = np.empty(len(x))
    for k in range(len(x)):
        xp, xm = x.copy(), x.copy()
        xp[k] += h
        xm[k] -= h
        g[k] = (f(xp) - f(xm)) / (2 * h)
    return g


def _fp32_point(rng, d):
    return rng.uniform(0.1, 0.9, d).astype(np.float32).astype(np.float64)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_posterior_gradients_match_central_differences(seed):
    fp, _, rng = _problem(seed)
    for _ in range(4):
        x = _fp32_point(rng, fp.X.shape[1])
        for t in range(2):
            m, v, dm, dv = opl.posterior_grad(fp, t, x)
            mc = lambda xx: opl.posterior(fp, np.asarray(xx, np.float32)[None])[0][0, t]
            vc = lambda xx: opl.posterior(fp, np.asarray(xx, np.float32)[None])[1][0, t]
            assert m == pytest.approx(mc(x), rel=1e-12, abs=1e-14)
            assert v == pytest.approx(vc(x), rel=1e-10, abs=1e-14)
            np.testing.assert_allclose(dm, _fd(mc, x, H), rtol=1e-5, atol=1e-8)
            np.testing.assert_allclose(dv, _fd(vc, x, H), rtol=1e-5, atol=1e-8)


def test_hvi_and_its_gradient():
    rng = np.random.default_rng(5)
    front = np.array([[0.1, 0.9], [0.3, 0.6], [0.5, 0.45], [0.8, 0.2]])
    ref = np.array([1.2, 1.2])
    for _ in range(20):
        y = rng.uniform(-0.2, 1.3, 2)
        v, g = opl.hvi2_grad(front, ref, y)
        assert v == pytest.approx(oracle.hvi(front, ref, y), abs=1e-14)
        fd = _fd(lambda yy: oracle.hvi(front, ref, yy), y, 1e-7)
        np.testing.assert_allclose(g, fd, atol=1e-6)


@pytest.mark.parametrize("seed", [3, 4])
def test_acquisition_gradient_matches_central_differences(seed):
    fp, eps, rng = _problem(seed)
    f = lambda xx: _acq_c(fp, eps, xx)
    clean = 0
    for _ in range(12):
        x = _fp32_point(rng, fp.X.shape[1])
        v, g = opl.mc_hvi_value_grad(fp, x, eps)
        assert v == pytest.approx(f(x), rel=1e-9, abs=1e-12)
        g1, g2 = _fd(f, x, H), _fd(f, x, H / 2)
        if np.abs(g1 - g2).max() > 1e-6 * max(1.0, np.abs(g1).max()):
            continue  # a draw crosses a strip edge within the step
        np.testing.assert_allclose(g, g1, rtol=2e-5, atol=1e-7)
        clean += 1
    assert clean >= 6


def test_optimiser_reaches_the_grid_maximum_in_one_dimension():
    rng = np.random.default_rng(7)
    X = rng.random((8, 1))
    Y = np.stack([(X[:, 0] - 0.2) ** 2, (X[:, 0] - 0.8) ** 2], 1)
    fp = opl.fit_problem(X, Y, np.full((2, 1), 0.3), np.ones(2), np.full(2, 1e-4),
                         np.array([1.5, 1.5]))
    eps = rng.standard_normal((2, 16)).astype(np.float32).astype(np.float64)
    grid = np.linspace(0.0, 1.0, 2001)
    vals = np.array([opl.mc_hvi_value_grad(fp, np.array([g]), eps)[0] for g in grid])
    starts = np.array([[0.05], [0.35], [0.5], [0.65], [0.95]])
    Xf, af = opl.optimize_acq(fp, starts, eps, np.zeros(1), np.ones(1), steps=300, lr=0.01)
    a0 = np.array([opl.mc_hvi_value_grad(fp, s, eps)[0] for s in starts])
    assert (af >= a0 - 1e-12).all()
    # the best start ends at the global maximum of the grid (to its resolution)
    assert af.max() >= vals.max() - 1e-4 * vals.max()
    # every end point is a local maximum of the grid values around it
    for xf, a in zip(Xf[:, 0], af):
        i = int(np.argmin(np.abs(grid - xf)))
        lo, hi = max(0, i - 20), min(len(grid), i + 21)
        assert a >= vals[lo:hi].max() - 1e-3 * vals.max()

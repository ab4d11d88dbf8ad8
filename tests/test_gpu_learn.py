"""Hyperparameter learning by maximising the log marginal likelihood (Sec. 6)
on the CUDA path against the oracle: the likelihood and its gradient at given
parameters (shared-memory and global-memory workspaces), and whole Adam
trajectories with several restarts per problem and objective. Both sides
compute in fp64, so the tolerances are those of fp64 rounding through a
factorisation of condition number up to about 1e6."""
import numpy as np
import pytest

import oracle
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _problem(wi, B, n, R, seed=0):
    w = wl.scaled(wl.WORKLOADS[wi], B=B, n=n)
    X = np.stack([wl.training_set(w, b)[0] for b in range(w.B)])
    Y = np.stack([wl.training_set(w, b)[1] for b in range(w.B)])
    Ys = np.stack([oracle.standardize(Y[b]) for b in range(w.B)])
    ls, s2, nz = wl.hyperparameters(w, 0)
    base = np.r_[np.log(ls[0]), np.log(s2[0]), np.log(10 * nz[0])]  # noise from 1e-3
    rng = np.random.default_rng(seed)
    theta0 = base + rng.normal(0.0, 0.5, (w.B, w.m, R, w.d + 2))
    return w, X, Ys, theta0


def _gpu(X, Ys, theta0, iters, lr):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    t = lambda a: torch.as_tensor(np.ascontiguousarray(a), dtype=torch.float64, device="cuda")
    th0 = t(theta0)
    theta = torch.empty_like(th0)
    grad = torch.empty_like(th0)
    mll = torch.empty(theta0.shape[:3], dtype=torch.float64, device="cuda")
    bt.boute_gp_learn(t(X), t(Ys), th0, iters, lr, theta, mll, grad)
    torch.cuda.synchronize()
    return theta.cpu().numpy(), mll.cpu().numpy(), grad.cpu().numpy()


@pytest.mark.parametrize("wi,B,n,R", [(0, 1, 32, 3), (1, 1, 128, 3), (4, 2, 200, 2)],
                         ids=["n32", "n128", "n200-global-workspace"])
def test_likelihood_and_gradient_match_oracle(wi, B, n, R):
    w, X, Ys, theta0 = _problem(wi, B, n, R)
    theta, mll, grad = _gpu(X, Ys, theta0, 0, 0.05)
    d = w.d
    for b in range(w.B):
        for t in range(w.m):
            for r in range(R):
                th = theta0[b, t, r]
                np.testing.assert_array_equal(theta[b, t, r], th)  # inside the bounds
                v, g = oracle.gp_mll(X[b], Ys[b][:, t], np.exp(th[:d]), np.exp(th[d]),
                                     np.exp(th[d + 1]), grad=True)
                assert mll[b, t, r] == pytest.approx(v, rel=1e-10, abs=1e-9)
                np.testing.assert_allclose(grad[b, t, r], g, rtol=1e-7,
                                           atol=1e-9 * np.abs(g).max())


@pytest.mark.parametrize("wi,B,n,R,iters", [(0, 1, 32, 4, 80), (1, 1, 128, 2, 40),
                                            (4, 1, 200, 1, 15)],
                         ids=["n32", "n128", "n200-global-workspace"])
def test_adam_trajectories_match_oracle(wi, B, n, R, iters):
    w, X, Ys, theta0 = _problem(wi, B, n, R, seed=1)
    lr = 0.05
    theta, mll, grad = _gpu(X, Ys, theta0, iters, lr)
    for b in range(w.B):
        for t in range(w.m):
            th_o, mll_o, g_o = oracle.gp_learn(X[b], Ys[b][:, t], theta0[b, t], iters, lr,
                                               grad=True)
            np.testing.assert_allclose(theta[b, t], th_o, rtol=0, atol=1e-7)
            np.testing.assert_allclose(mll[b, t], mll_o, rtol=1e-9, atol=1e-8)
            # the learner climbs: the end is above the start
            for r in range(R):
                th = theta0[b, t, r]
                d = w.d
                v0 = oracle.gp_mll(X[b], Ys[b][:, t], np.exp(np.clip(th[:d], -6.9, 6.9)),
                                   np.exp(np.clip(th[d], -6.9, 6.9)),
                                   np.exp(np.clip(th[d + 1], -9.2, 2.3)))
                assert mll[b, t, r] > v0


def test_invalid_arguments():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    X = torch.zeros((1, 8, 2), dtype=torch.float64, device="cuda")
    Ys = torch.zeros((1, 8, 2), dtype=torch.float64, device="cuda")
    th = torch.zeros((1, 2, 1, 4), dtype=torch.float64, device="cuda")
    mll = torch.zeros((1, 2, 1), dtype=torch.float64, device="cuda")
    with pytest.raises(bt.BouteError):
        bt.boute_gp_learn(X, Ys, th, -1, 0.1, th.clone(), mll)
    with pytest.raises(bt.BouteError):
        bt.boute_gp_learn(X, Ys, th, 5, float("nan"), th.clone(), mll)


# ---- the composite kernel's learner ---------------------------------------------
def _composite_problem(wi, n, R, seed=2):
    w = wl.composite(wl.scaled(wl.WORKLOADS[wi], B=1, n=n))
    X, Y = wl.training_set(w, 0)
    Ys = oracle.standardize(oracle.outcome_transform(Y, list(w.transforms)))
    dtau, kc = wl.kernel_params(w, 0)
    ls, s2, nz = wl.hyperparameters(w, 0)
    base = np.r_[np.log(ls[0]), np.log(s2[0]), np.log(1e-3), np.log(kc[0, 0]), np.log(kc[0, 1]),
                 kc[0, 2]]
    rng = np.random.default_rng(seed)
    theta0 = base + rng.normal(0.0, 0.3, (1, w.m, R, w.d + 5))
    pref = kc[None, :, 3:]  # B x m x (d - dtau)
    return w, X[None], Ys[None], theta0, dtau, pref


def _gpu_k(X, Ys, dtau, pref, theta0, iters, lr):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    t = lambda a: torch.as_tensor(np.ascontiguousarray(a), dtype=torch.float64, device="cuda")
    th0 = t(theta0)
    theta = torch.empty_like(th0)
    grad = torch.empty_like(th0)
    mll = torch.empty(theta0.shape[:3], dtype=torch.float64, device="cuda")
    bt.boute_gp_learn_k(t(X), t(Ys), dtau, t(pref), th0, iters, lr, theta, mll, grad)
    torch.cuda.synchronize()
    return theta.cpu().numpy(), mll.cpu().numpy(), grad.cpu().numpy()


@pytest.mark.parametrize("wi,n,R", [(1, 128, 2), (2, 200, 1)], ids=["n128", "n200-global"])
def test_composite_likelihood_gradient_and_trajectory_match_oracle(wi, n, R):
    w, X, Ys, theta0, dtau, pref = _composite_problem(wi, n, R)
    d = w.d
    theta, mll, grad = _gpu_k(X, Ys, dtau, pref, theta0, 0, 0.05)
    for t in range(w.m):
        for r in range(R):
            th = theta0[0, t, r]
            kc = np.concatenate([[np.exp(th[d + 2]), np.exp(th[d + 3]), th[d + 4]], pref[0, t]])
            v, g = oracle.gp_mll(X[0], Ys[0][:, t], np.exp(th[:d]), np.exp(th[d]),
                                 np.exp(th[d + 1]), grad=True, kernel=(dtau, kc))
            assert mll[0, t, r] == pytest.approx(v, rel=1e-10, abs=1e-9)
            np.testing.assert_allclose(grad[0, t, r], g, rtol=1e-7, atol=1e-9 * np.abs(g).max())
    iters, lr = 12, 0.05
    theta, mll, _ = _gpu_k(X, Ys, dtau, pref, theta0, iters, lr)
    for t in range(w.m):
        th_o, mll_o = oracle.gp_learn(X[0], Ys[0][:, t], theta0[0, t], iters, lr,
                                      kernel=(dtau, pref[0, t]))
        np.testing.assert_allclose(theta[0, t], th_o, rtol=0, atol=1e-7)
        np.testing.assert_allclose(mll[0, t], mll_o, rtol=1e-9, atol=1e-8)

"""The optimisation loop (Sec. 5.2 "Overall MOBO workflow" (i)-(iii), stopped
by the stability rule of Sec. 7) on the GPU against the oracle: every
iteration's choice must be a best candidate of the oracle's acquisition on
the same observations and hyperparameters, the learned hyperparameters must
be the oracle learner's from the same start, the observations must be the
objective at the chosen candidates, and the loop must stop exactly when the
observed Pareto set has been stable for `patience` iterations."""
import numpy as np
import pytest

import oracle
from oracle import pipeline as opl

pytestmark = pytest.mark.gpu


def _objective(x):
    d = x.size
    return np.array([((x - 0.25) ** 2).sum() / d, ((x - 0.75) ** 2).sum() / d])


def _objective_lq(x):
    """Latency and quality of a routing (x[:2]) + deployment (x[2:], GPU
    counts) configuration."""
    xh = x.copy()
    xh[2:] /= 4.0
    f1, f2 = _objective(xh)
    return np.array([np.exp(f1), 1.0 / (1.0 + np.exp(4.0 * f2 - 0.5))])


def _pareto_set(Y, codes=None):
    Z = Y if codes is None else oracle.outcome_transform(Y, codes)
    mask, _ = oracle.pareto_front(Z, np.full(Y.shape[1], np.inf))
    return set(np.flatnonzero(mask).tolist())


def _check_run(res, cand, n0, patience, max_evals, mode, eps, ls0, s2, noise, learn,
               objective=_objective, codes=None, comp=None):
    """comp: (d_tau, kc0) of the composite kernel, else None."""
    X, Y, sel, theta = res["X"], res["Y"], res["sel"], res["theta"]
    n = len(X)
    assert n == n0 + len(sel)
    ref = np.array([1.1, 1.1])
    d = cand.shape[1]
    th_prev = np.concatenate([np.log(ls0), np.log(s2)[:, None], np.log(noise)[:, None]], 1)
    if comp:
        kc0 = comp[1]
        th_prev = np.concatenate([th_prev, np.log(kc0[:, :2]), kc0[:, 2:3]], 1)
    for t, pick in enumerate(sel):
        nt = n0 + t
        np.testing.assert_array_equal(X[nt], cand[pick].astype(np.float64))
        np.testing.assert_array_equal(Y[nt], objective(X[nt]))
        th = theta[t]
        if learn:  # the oracle learner from the previous iteration's parameters
            Z = Y[:nt] if codes is None else oracle.outcome_transform(Y[:nt], codes)
            ys = oracle.standardize(Z)
            for obj in range(2):
                kern = None if comp is None else (comp[0], comp[1][obj, 3:])
                th_o, mll_o = oracle.gp_learn(X[:nt], ys[:, obj], th_prev[obj][None], learn[0],
                                              learn[1], kernel=kern)
                np.testing.assert_allclose(th[obj], th_o[0], rtol=0, atol=1e-6)
        else:
            np.testing.assert_allclose(th, th_prev, rtol=0, atol=0)
        th_prev = th
        kernel = None
        if comp:
            kc_t = np.concatenate([np.exp(th[:, d + 2:d + 4]), th[:, d + 4:d + 5], comp[1][:, 3:]], 1)
            kernel = (comp[0], kc_t)
        fp = opl.fit_problem(X[:nt], Y[:nt], np.exp(th[:, :d]), np.exp(th[:, d]),
                             np.exp(th[:, d + 1]), ref, kernel=kernel, transforms=codes)
        mean, var = opl.posterior(fp, cand)
        acq = opl.acquisition(fp, mean, var, mode, eps)
        best = acq.max()
        assert acq[pick] >= best - 1e-3 * max(abs(best), 1e-6), (t, acq[pick], best)
    # stopping rule
    sets = [_pareto_set(Y[:k], codes) for k in range(n0, n + 1)]
    stable = 0
    for k in range(1, len(sets)):
        stable = stable + 1 if sets[k] == sets[k - 1] else 0
        if k < len(sets) - 1:
            assert stable < patience  # it would have stopped here
    assert res["converged"] == (stable >= patience)
    if not res["converged"]:
        assert n == max_evals


@pytest.mark.parametrize("learn", [None, (15, 0.05)], ids=["fixed", "learned"])
def test_loop_choices_match_oracle(learn):
    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(7)
    d, N, n0 = 4, 1536, 6
    cand = rng.random((N, d)).astype(np.float32)
    X0 = cand[:n0].astype(np.float64)
    Y0 = np.stack([_objective(x) for x in X0])
    ls0 = np.full((2, d), 0.4)
    s2, noise = np.ones(2), np.full(2, 1e-4)
    mode = "mc" if learn else "ehvi"
    S = 128
    # Monte-Carlo: the engine's own normals from a seed, regenerated here by
    # the oracle's implementation of the same generator
    eps = oracle.base_normals(31, 1, N, 2, S)[0] if mode == "mc" else None
    max_evals, patience = 24, 4
    res = bt.boute_mobo_run(_objective, cand, [1.1, 1.1], ls0, s2, noise, X0, Y0,
                            mode=bt.BOUTE_ACQ_MC_HVI if mode == "mc" else bt.BOUTE_ACQ_EHVI2D,
                            S=S if mode == "mc" else 0, eps=None, seed=31, max_evals=max_evals,
                            patience=patience, learn_iters=learn[0] if learn else 0,
                            learn_lr=learn[1] if learn else 0.05)
    assert len(res["sel"]) >= patience  # converged (stable that long) or ran out of budget
    _check_run(res, cand, n0, patience, max_evals, mode, eps, ls0, s2, noise, learn)
    # the loop improves the observed front: its hypervolume never falls
    hv = [oracle.hv(Y[list(_pareto_set(Y))], np.array([1.0, 1.0]))
          for Y in (res["Y"][:k] for k in range(n0, len(res["Y"]) + 1))]
    assert all(b >= a - 1e-12 for a, b in zip(hv, hv[1:]))


def test_loop_with_composite_kernel_transforms_and_learning():
    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(9)
    N, n0, dtau = 1024, 8, 2
    cand = np.concatenate([rng.random((N, 2)), rng.integers(0, 5, (N, 2))], 1).astype(np.float32)
    X0 = cand[:n0].astype(np.float64)
    Y0 = np.stack([_objective_lq(x) for x in X0])
    ls0 = np.tile([0.4, 0.4, 1.6, 1.6], (2, 1))
    s2, noise = np.ones(2), np.full(2, 1e-3)
    kc0 = np.concatenate([np.tile([0.5, 0.1, 0.05], (2, 1)), rng.random((2, 2))], 1)
    codes = [bt.BOUTE_TF_LOG, bt.BOUTE_TF_LOGIT | bt.BOUTE_TF_NEGATE]
    learn = (10, 0.05)
    max_evals, patience = 20, 4
    res = bt.boute_mobo_run(_objective_lq, cand, [1.1, 1.1], ls0, s2, noise, X0, Y0,
                            max_evals=max_evals, patience=patience, learn_iters=learn[0],
                            learn_lr=learn[1], transforms=codes, d_tau=dtau, kc=kc0)
    assert len(res["sel"]) >= patience
    _check_run(res, cand, n0, patience, max_evals, "ehvi", None, ls0, s2, noise, learn,
               objective=_objective_lq, codes=codes, comp=(dtau, kc0))
    assert res["theta"].shape[2] == cand.shape[1] + 5


def test_objective_errors_stop_the_loop():
    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(8)
    cand = rng.random((256, 3)).astype(np.float32)
    X0 = cand[:4].astype(np.float64)
    Y0 = np.stack([_objective(x) for x in X0])

    def bad(x):
        raise ValueError("evaluation failed")

    with pytest.raises(ValueError):
        bt.boute_mobo_run(bad, cand, [1.1, 1.1], np.full((2, 3), 0.4), np.ones(2),
                          np.full(2, 1e-4), X0, Y0, max_evals=8, patience=3)


def test_loop_with_gradient_refinement():
    """Sec. 5.2 step (ii) with the acquisition optimised over the decision
    space: each iteration ascends from the pool's best candidates and
    evaluates the best end point. Against the oracle on the same
    observations: the end point's sample-average acquisition (the loop's
    shared normals, regenerated here) is at least its start's and matches the
    oracle's own ascent from that start."""
    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(13)
    d, N, n0, S = 3, 1024, 6, 32
    cand = rng.random((N, d)).astype(np.float32)
    X0 = cand[:n0].astype(np.float64)
    Y0 = np.stack([_objective(x) for x in X0])
    ls0 = np.full((2, d), 0.4)
    s2, noise = np.ones(2), np.full(2, 1e-4)
    seed, starts, steps, lr = 17, 4, 25, 0.02
    max_evals = n0 + 6
    res = bt.boute_mobo_run(_objective, cand, [1.1, 1.1], ls0, s2, noise, X0, Y0,
                            mode=bt.BOUTE_ACQ_MC_HVI, S=S, seed=seed, max_evals=max_evals,
                            patience=100, refine_starts=starts, refine_steps=steps, refine_lr=lr)
    X, Y, sel = res["X"], res["Y"], res["sel"]
    assert len(sel) == max_evals - n0
    er = oracle.base_normals(seed ^ 0xbb67ae8584caa73b, 1, 1, 2, S)[0, 0].astype(np.float64)
    for t, p in enumerate(sel):
        nt = n0 + t
        x = X[nt]
        assert (x >= 0).all() and (x <= 1).all()
        np.testing.assert_array_equal(Y[nt], _objective(x))
        fp = opl.fit_problem(X[:nt], Y[:nt], ls0, s2, noise, np.array([1.1, 1.1]))
        a_end = opl.mc_hvi_value_grad(fp, x, er)[0]
        a_start = opl.mc_hvi_value_grad(fp, cand[p].astype(np.float64), er)[0]
        _, ao = opl.optimize_acq(fp, cand[p][None].astype(np.float64), er, np.zeros(d),
                                 np.ones(d), steps, lr)
        scale = max(abs(ao[0]), abs(a_start), 1e-12)
        assert a_end >= a_start - 1e-5 * scale, (t, a_end, a_start)
        assert abs(a_end - ao[0]) <= 1e-3 * scale, (t, a_end, ao[0])

"""The paper's composite kernel (Sec. 5.2 "Additive kernels" with the
preference weighting of S5, as Sec. 6 assembles it: a Matern-5/2 kernel on
the routing features, a preference-weighted Matern-3/2 kernel on the
deployment features and their scaled product) and the Log / Logit outcome
transforms (S4) on the CUDA path against the oracle: the step-by-step calls
(the posterior builds K* itself), the engine (K* computed beside the fit) and
the return to the Matern-5/2 kernel.

Tolerances: the composite kernel's prior variance k(x, x) = s2 + s2_x +
s2_c w(x)^2 varies with the candidate, so the scale of the variance check is
its largest value and the mean is checked against the fp32 forward error
bound of the cross-covariance, 16 eps32 sum_j |K*_j alpha_j| (the additive
kernel's long deployment lengthscales make the mean cancel more than the
Matern-5/2 workloads do), plus 1e-5 of the prior standard deviation."""
import dataclasses

import numpy as np
import pytest

import oracle
from _pipeline import (ACQ_FLOOR, ACQ_REL, POST_REL, check_acq, check_topk_consistent_tol,
                       gpu_pipeline, host_problem, oracle_fit)
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

EPS32 = float(np.finfo(np.float32).eps)


def _variant(wi, N, B=1, n=None, d=None):
    base = wl.WORKLOADS[wi]
    if d is not None:
        base = dataclasses.replace(base, d=d, name=f"{base.name}-d{d}")
    return wl.composite(wl.scaled(base, N=N, B=B, n=n))


def _check_posterior(hp, b, mean_g, var_g, fp=None):
    """mean_g, var_g: m x N from the GPU; against the oracle's posterior."""
    fp = fp or oracle_fit(hp, b)
    mean, var = opl.posterior(fp, hp.Xc[b])
    m = hp.w.m
    for t in range(m):
        kern = (hp.d_tau, hp.kc[b][t])
        ls, s2 = hp.ls[b][t], hp.s2[b][t]
        Xc = hp.Xc[b].astype(np.float64)
        prior = np.array([oracle.kernel(c, c, ls, s2, kern) for c in Xc])
        Ks = np.array([[oracle.kernel(c, x, ls, s2, kern) for x in hp.X[b]] for c in Xc])
        bound = 16 * EPS32 * (np.abs(Ks) @ np.abs(fp.alpha[t])) + POST_REL * np.sqrt(prior.max())
        err_m = np.abs(mean_g[t] - mean[:, t])
        assert np.all(np.isfinite(mean_g[t]))
        assert np.all(err_m <= bound), f"mean err {err_m.max():.3g} (objective {t})"
        err_v = np.abs(var_g[t] - var[:, t]) / prior.max()
        assert np.all(np.isfinite(var_g[t])) and np.all(var_g[t] >= 0)
        assert err_v.max() <= POST_REL, f"var rel err {err_v.max():.3g} (objective {t})"
        assert prior.max() > prior.min() * 1.05, "the preference weights vary too little"
    return mean, var


CASES = [  # (workload, N, B, n, d)
    (1, 2000 + 13, 1, None, None),   # d 12: 6 routing + 6 deployment features
    (0, 1000 + 1, 1, None, None),    # d 6, n 32
    (2, 1500, 1, 200, None),         # d 16, n 200: the fit's global-memory path
    (3, 700, 1, 96, None),           # d 24, m 3
    (4, 900, 3, 64, None),           # batched problems, per-problem preferences
    (0, 600, 1, 48, 32),             # d 32
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"w{c[0]}-N{c[1]}-B{c[2]}-n{c[3]}-d{c[4]}")
def test_composite_posterior_step_by_step_matches_oracle(case):
    wi, N, B, n, d = case
    w = _variant(wi, N, B, n, d)
    hp = host_problem(w)
    g = gpu_pipeline(hp)
    assert g["status"] == 0
    for b in range(w.B):
        fp = oracle_fit(hp, b)
        np.testing.assert_allclose(g["Ys"][b], fp.Ys, rtol=0, atol=1e-12)
        assert g["mask"][b].tolist() == fp.mask.tolist()
        _check_posterior(hp, b, g["mean"][b], g["var"][b], fp)


def test_outcome_transforms_in_standardize():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(3)
    Y = np.stack([np.exp(rng.normal(0, 1, (2, 50))), rng.uniform(0.02, 0.98, (2, 50)),
                  rng.normal(0, 2, (2, 50))], 2)
    codes = [bt.BOUTE_TF_LOG, bt.BOUTE_TF_LOGIT | bt.BOUTE_TF_NEGATE, bt.BOUTE_TF_IDENTITY]
    Yd = torch.as_tensor(Y, device="cuda")
    Ys = torch.empty_like(Yd)
    bt.boute_standardize(Yd, Ys, transforms=codes)
    got = Ys.cpu().numpy()
    for b in range(2):
        want = oracle.standardize(oracle.outcome_transform(Y[b], codes))
        np.testing.assert_allclose(got[b], want, rtol=0, atol=1e-12)
    with pytest.raises(bt.BouteError):
        bt.boute_standardize(Yd, Ys, transforms=[3, 0, 0])


def _engine_scores(e, w, inputs):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device="cuda")
    val = torch.empty((w.B, w.k), dtype=torch.float32, device="cuda")
    bt.boute_engine_step(e, *inputs, idx, val)
    acq = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
    mean = torch.empty((w.B, w.m, w.N), dtype=torch.float32, device="cuda")
    var = torch.empty_like(mean)
    bt.boute_engine_scores(e, acq=acq, mean=mean, var=var)
    return dict(idx=idx.cpu().numpy(), val=val.cpu().numpy(), acq=acq.cpu().numpy(),
                mean=mean.cpu().numpy(), var=var.cpu().numpy())


@pytest.mark.parametrize("wi,N,B", [(1, 3000 + 5, 1), (0, 4096 + 77, 1), (4, 1500 + 1, 3)],
                         ids=["mc2-fused-selection", "ehvi", "ehvi-batched"])
def test_composite_engine_steps(wi, N, B):
    import torch
    from test_gpu_engine import _dev, _engine

    from paper_2602_10729_gb300 import boute as bt
    w = _variant(wi, N, B, n=None if wi != 4 else 96)
    hp = host_problem(w)
    plain = dataclasses.replace(hp, d_tau=0, kc=None, transforms=())
    e = _engine(w)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        s0 = _engine_scores(e, w, _dev(hp))  # Matern-5/2, raw outcomes
        bt.boute_engine_set_kernel(e, hp.d_tau, hp.kc)
        bt.boute_engine_set_outcome_transforms(e, list(hp.transforms))
        s1 = _engine_scores(e, w, _dev(hp))
        s1b = _engine_scores(e, w, _dev(hp))  # graph replay
        bt.boute_engine_set_kernel(e, 0, None)
        bt.boute_engine_set_outcome_transforms(e, None)
        s2 = _engine_scores(e, w, _dev(hp))
    e.free()
    for key in s0:
        assert np.array_equal(s2[key], s0[key]), key
        assert np.array_equal(s1b[key], s1[key]), key
    # the Matern-5/2 steps are the plain problem's steps
    g0 = gpu_pipeline(plain)
    np.testing.assert_array_equal(s0["acq"], g0["acq"])
    # the composite steps against the step-by-step calls and the oracle
    g = gpu_pipeline(hp)
    for b in range(w.B):
        np.testing.assert_allclose(s1["mean"][b], g["mean"][b], rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(s1["var"][b], g["var"][b], rtol=1e-6, atol=1e-6)
        fp = oracle_fit(hp, b)
        _check_posterior(hp, b, s1["mean"][b], s1["var"][b], fp)
        eps = None if hp.eps is None else hp.eps[b]
        want = opl.acquisition(fp, s1["mean"][b].T.astype(np.float64),
                               s1["var"][b].T.astype(np.float64), w.mode, eps)
        check_acq(s1["acq"][b], want)
        tol = ACQ_REL * np.maximum(np.abs(want), ACQ_FLOOR * np.abs(want).max())
        check_topk_consistent_tol(s1["idx"][b], want, w.k, tol)
        assert np.array_equal(s1["val"][b], s1["acq"][b][s1["idx"][b]])


@pytest.mark.parametrize("dtau", [0, 6], ids=["all-deployment", "all-routing"])
def test_composite_degenerate_splits(dtau):
    """d_tau = 0 (no routing features: k = s2 + s2_c w w* k32 + s2_x k32) and
    d_tau = d (no deployment features: k = (s2 + s2_x) k52 + s2_c)."""
    w = dataclasses.replace(_variant(0, 777, 1, 40), d_tau=dtau)
    hp = host_problem(w)
    dc = w.d - dtau
    rng = np.random.default_rng(12)
    hp = dataclasses.replace(hp, d_tau=dtau,
                             kc=np.concatenate([np.tile([0.5, 0.1, 0.05], (1, w.m, 1)),
                                                rng.random((1, w.m, dc))], 2))
    g = gpu_pipeline(hp)
    assert g["status"] == 0
    fp = oracle_fit(hp, 0)
    mean, var = opl.posterior(fp, hp.Xc[0])
    for t in range(w.m):
        kern = (hp.d_tau, hp.kc[0][t])
        prior = np.array([oracle.kernel(c, c, hp.ls[0][t], hp.s2[0][t], kern)
                          for c in hp.Xc[0].astype(np.float64)])
        Ks = np.array([[oracle.kernel(c, x, hp.ls[0][t], hp.s2[0][t], kern) for x in hp.X[0]]
                       for c in hp.Xc[0].astype(np.float64)])
        bound = 16 * EPS32 * (np.abs(Ks) @ np.abs(fp.alpha[t])) + POST_REL * np.sqrt(prior.max())
        assert np.all(np.abs(g["mean"][0, t] - mean[:, t]) <= bound)
        assert np.abs(g["var"][0, t] - var[:, t]).max() <= POST_REL * prior.max()

"""Constrained acquisition (Sec. 5.2, constrained qNEHVI: the hypervolume
improvement times the indicator that every objective meets its threshold) on
the CUDA path against the oracle: the closed-form 2-objective EHVI, the
Monte-Carlo estimate for m = 2 and 3 on the vectorised (S = 128) and scalar
sample paths, the selecting acquisition kernel inside the engine, and the
engine's switch back to the unconstrained acquisition.

The Monte-Carlo cases place each threshold in a gap between the sample values
of its objective, wider than the fp32 error of a sample, so that the kernel
(fp32) and the oracle (fp64) make the same feasibility decision for every
sample; the estimates then differ by rounding alone."""
import numpy as np
import pytest

import oracle
from _pipeline import (ACQ_FLOOR, ACQ_REL, check_acq, check_topk_consistent_tol, gpu_pipeline,
                       host_problem, oracle_fit)
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

INF = np.inf


def _posterior32(hp):
    """Oracle posterior of every problem rounded to fp32: B x m x N each."""
    ms, vs = [], []
    for b in range(hp.w.B):
        mean, var = opl.posterior(oracle_fit(hp, b), hp.Xc[b])
        ms.append(mean.T.astype(np.float32))
        vs.append(var.T.astype(np.float32))
    return np.stack(ms), np.stack(vs)


def _gap_threshold(y, q, margin=1e-5):
    """A threshold near the q-quantile of the sample values y whose distance
    to every sample exceeds margin * max(1, |threshold|)."""
    v = np.sort(np.asarray(y, np.float64).ravel())
    i = int(q * (len(v) - 1))
    lo, hi = max(i - 2000, 1), min(i + 2000, len(v) - 1)
    gaps = v[lo:hi + 1] - v[lo - 1:hi]
    j = int(np.argmax(gaps))
    c = 0.5 * (v[lo - 1 + j] + v[lo + j])
    assert gaps[j] / 2 > margin * max(1.0, abs(c)), "no clear gap near the quantile"
    return c


def _samples(mean, var, eps, t):
    """Sample values of objective t: mean, var: m x N (fp32), eps: N x m x S."""
    sg = np.sqrt(var[t].astype(np.float64))
    return mean[t].astype(np.float64)[:, None] + sg[:, None] * eps[:, t, :].astype(np.float64)


def _mc_thresholds(mean, var, eps, qs):
    """One gap threshold per objective (q = None: unconstrained)."""
    return np.array([INF if q is None else _gap_threshold(_samples(mean, var, eps, t), q)
                     for t, q in enumerate(qs)])


# ---- closed-form EHVI -------------------------------------------------------------
@pytest.mark.parametrize("cons", [
    [(0.0, 0.3), (INF, -0.2), (-0.4, INF)],
    [(-1.0, -1.0), (0.8, 0.8), (1.5, 1.5)],
], ids=["mixed", "tight-loose-beyond-ref"])
def test_constrained_ehvi_matches_oracle(cons):
    w = wl.scaled(wl.WORKLOADS[4], N=3001, B=3)
    hp = host_problem(w)
    mean, var = _posterior32(hp)
    var[:, :, :40] = 0.0  # candidates without uncertainty: the indicator is a step
    cons = np.array(cons, np.float64)
    g = gpu_pipeline(hp, mean_var_in=(mean, var), cons=cons)
    assert g["status"] == 0
    for b in range(w.B):
        fp = oracle_fit(hp, b)
        want = oracle.ehvi2d(mean[b].T.astype(np.float64), var[b].T.astype(np.float64), fp.front,
                             fp.ref, cons=cons[b])
        check_acq(g["acq"][b], want)


def test_thresholds_beyond_ref_leave_ehvi_unchanged():
    # samples above the reference point improve nothing, so thresholds at or
    # beyond it constrain nothing
    w = wl.scaled(wl.WORKLOADS[4], N=2000, B=2)
    hp = host_problem(w)
    mean, var = _posterior32(hp)
    g0 = gpu_pipeline(hp, mean_var_in=(mean, var))
    g1 = gpu_pipeline(hp, mean_var_in=(mean, var), cons=np.array(hp.ref) + 0.5)
    for b in range(w.B):
        check_acq(g1["acq"][b], g0["acq"][b].astype(np.float64))


# ---- Monte-Carlo ------------------------------------------------------------------
MC_CASES = [  # (workload, S, quantiles per objective)
    (1, 128, (0.55, 0.7)),
    (1, 50, (0.3, None)),
    (1, 128, (None, 0.4)),
    (3, 128, (0.6, 0.75, 0.9)),
    (3, 40, (0.5, None, 0.6)),
]


@pytest.mark.parametrize("case", MC_CASES, ids=lambda c: f"m{wl.WORKLOADS[c[0]].m}-S{c[1]}-{c[2]}")
def test_constrained_mc_hvi_matches_oracle(case):
    wi, S, qs = case
    w = wl.scaled(wl.WORKLOADS[wi], N=1203, B=1, n=96, S=S)
    hp = host_problem(w)
    mean, var = _posterior32(hp)
    cons = _mc_thresholds(mean[0], var[0], hp.eps[0], qs)[None]
    g = gpu_pipeline(hp, mean_var_in=(mean, var), cons=cons)
    assert g["status"] == 0
    fp = oracle_fit(hp, 0)
    want = oracle.mc_hvi(mean[0].T.astype(np.float64), var[0].T.astype(np.float64), hp.eps[0],
                         fp.front, fp.ref, cons=cons[0])
    check_acq(g["acq"][0], want)
    # the constraint removes improvement: never above the unconstrained value
    want0 = oracle.mc_hvi(mean[0].T.astype(np.float64), var[0].T.astype(np.float64), hp.eps[0],
                          fp.front, fp.ref)
    assert np.all(want <= want0 + 1e-12)
    assert (want < want0 - 1e-9).any(), "the thresholds constrain nothing"


@pytest.mark.parametrize("wi,S", [(4, 0), (1, 128), (1, 50), (3, 128), (3, 40)])
def test_infinite_thresholds_reproduce_the_unconstrained_kernels(wi, S):
    base = wl.WORKLOADS[wi]
    w = wl.scaled(base, N=1500, B=min(base.B, 2), n=96, S=S if base.mode == "mc" else None)
    hp = host_problem(w)
    mean, var = _posterior32(hp)
    g0 = gpu_pipeline(hp, mean_var_in=(mean, var))
    g1 = gpu_pipeline(hp, mean_var_in=(mean, var), cons=np.full((w.B, w.m), INF))
    assert np.array_equal(g0["acq"], g1["acq"])


# ---- the engine ---------------------------------------------------------------------
def _engine_step(e, w, dev_inputs, host_inputs=None):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device="cuda")
    val = torch.empty((w.B, w.k), dtype=torch.float32, device="cuda")
    bt.boute_engine_step(e, *dev_inputs, idx, val)
    acq = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
    mean = torch.empty((w.B, w.m, w.N), dtype=torch.float32, device="cuda")
    var = torch.empty_like(mean)
    bt.boute_engine_scores(e, acq=acq, mean=mean, var=var)
    out = dict(idx=idx.cpu().numpy(), val=val.cpu().numpy(), acq=acq.cpu().numpy(),
               mean=mean.cpu().numpy(), var=var.cpu().numpy())
    if host_inputs is not None:
        hi = torch.empty((w.B, w.k), dtype=torch.int64).pin_memory()
        hv = torch.empty((w.B, w.k), dtype=torch.float32).pin_memory()
        bt.boute_engine_step_host(e, *host_inputs, hi, hv)
        out.update(host_idx=hi.numpy().copy(), host_val=hv.numpy().copy())
    return out


@pytest.mark.parametrize("wi,N,B", [(1, 3000 + 5, 1), (0, 4096 + 77, 1), (4, 1500 + 1, 3)],
                         ids=["mc2-fused-selection", "ehvi", "ehvi-batched"])
def test_engine_constrained_steps(wi, N, B):
    import torch
    from test_gpu_engine import _dev, _engine, _host

    from paper_2602_10729_gb300 import boute as bt
    w = wl.scaled(wl.WORKLOADS[wi], N=N, B=B)
    hp = host_problem(w)
    e = _engine(w)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        s0 = _engine_step(e, w, _dev(hp))
        if w.mode == "mc":
            cons = np.stack([_mc_thresholds(s0["mean"][b], s0["var"][b], hp.eps[b], (0.5, 0.65))
                             for b in range(w.B)])
        else:
            cons = np.array([[0.1, 0.4], [INF, -0.3], [-0.5, 0.6]][:w.B], np.float64)
        bt.boute_engine_set_constraints(e, torch.as_tensor(cons))
        s1 = _engine_step(e, w, _dev(hp), _host(hp))
        bt.boute_engine_set_constraints(e, None)
        s2 = _engine_step(e, w, _dev(hp))
    e.free()
    # the posterior is the same in every step; switching back restores the
    # unconstrained step exactly
    assert np.array_equal(s1["mean"], s0["mean"]) and np.array_equal(s1["var"], s0["var"])
    for key in ("acq", "idx", "val"):
        assert np.array_equal(s2[key], s0[key]), key
    assert np.array_equal(s1["host_idx"], s1["idx"]) and np.array_equal(s1["host_val"], s1["val"])
    assert not np.array_equal(s1["acq"], s0["acq"])
    for b in range(w.B):
        fp = oracle_fit(hp, b)
        eps = None if hp.eps is None else hp.eps[b]
        want = opl.acquisition(fp, s1["mean"][b].T.astype(np.float64),
                               s1["var"][b].T.astype(np.float64), w.mode, eps, cons=cons[b])
        check_acq(s1["acq"][b], want)
        tol = ACQ_REL * np.maximum(np.abs(want), ACQ_FLOOR * np.abs(want).max())
        check_topk_consistent_tol(s1["idx"][b], want, w.k, tol)
        assert np.array_equal(s1["val"][b], s1["acq"][b][s1["idx"][b]])

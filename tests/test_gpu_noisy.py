"""The noisy acquisition (Sec. 5.2, constrained qNEHVI over the joint
posterior of the observed points and the candidate) through the C-ABI
against the oracle, element by element:

* the in-sample draws, and the joint posterior's mean, conditional variance
  and shifts, within the posterior tolerance (1e-5 of the prior scale);
* each draw's front, bit-exact against the oracle's front of the GPU's own
  draws (the same fp32 values decide membership on both sides);
* the acquisition kernel against the oracle acquisition of the GPU's
  intermediates (1e-4);
* the whole chain against the oracle's own chain, allowing for the
  posterior tolerance's effect on the acquisition, and the selection;
* a handle with in-sample draws still gives the plain posterior, and shapes
  beyond the limits are refused."""
import dataclasses

import numpy as np
import pytest

import oracle
from _pipeline import (ACQ_FLOOR, ACQ_REL, POST_REL, check_acq, check_mean, check_topk_consistent_tol,
                       host_problem, oracle_fit)
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

# (workload, N, n, S, B, constrained): several tiles and a ragged tail; S not a
# multiple of 128 (a partial G block) and above 128 (two G blocks); n not a
# multiple of 32; a batch of problems; the composite kernel
CASES = [
    (1, 3000 + 77, 128, 128, 1, False),
    (1, 2048 + 5, 100, 40, 1, True),
    (4, 1500 + 3, 32, 200, 2, False),
    (4, 999, 64, 64, 3, True),
]


def _workload(wi, N, n, S, B, comp=False):
    w = wl.WORKLOADS[wi]
    if comp:
        w = wl.composite(w)
    w = wl.scaled(w, N=N, B=B, n=n)
    return dataclasses.replace(w, mode="mc", S=S, k=min(16, N))


def _cons(hp):
    """Thresholds that cut some of the observed front (standardised units)."""
    return np.tile([0.2, 0.4], (hp.w.B, 1))


def _gpu(hp, z, cons):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = hp.w
    B, n, d, m, S, N = w.B, w.n, w.d, w.m, w.S, hp.Xc.shape[1]
    dev = torch.device("cuda")
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), device=dev, dtype=dt)
    f64, f32 = torch.float64, torch.float32
    X, Y = t(hp.X, f64), t(hp.Y, f64)
    ls, s2, nz, ref = t(hp.ls, f64), t(hp.s2, f64), t(hp.noise, f64), t(hp.ref, f64)
    Xc, eps, zt = t(hp.Xc, f32), t(hp.eps, f32), t(z, f32)
    cn = None if cons is None else t(cons, f64)
    Ys = torch.empty_like(Y)
    bt.boute_standardize(Y, Ys, transforms=hp.transforms or None)
    gp = bt.boute_gp_create(B, n, d, m)
    if hp.kc is not None:
        bt.boute_gp_set_kernel(gp, hp.d_tau, hp.kc)
    bt.boute_gp_set_insample(gp, S)
    bt.boute_gp_fit(gp, X, Ys, ls, s2, nz)
    Yin = torch.empty((B, m, S, n), dtype=f32, device=dev)
    bt.boute_gp_insample(gp, Ys, s2, nz, zt, Yin)
    assert bt.boute_gp_status(gp) == 0
    mean = torch.empty((B, m, N), dtype=f32, device=dev)
    cvar = torch.empty_like(mean)
    shift = torch.empty((B, m, S, N), dtype=f32, device=dev)
    bt.boute_gp_posterior_joint(gp, Xc, N, mean, cvar, shift)
    pm, pv = torch.empty_like(mean), torch.empty_like(mean)
    bt.boute_gp_posterior(gp, Xc, N, pm, pv)  # the plain posterior on the same handle
    strips = torch.empty((B, S, n + 1, 4), dtype=f32, device=dev)
    counts = torch.empty((B, S), dtype=torch.int32, device=dev)
    bt.boute_insample_fronts(Yin, B, n, S, ref, strips, counts, cons=cn)
    acq = torch.empty((B, N), dtype=f32, device=dev)
    bt.boute_acq_nehvi2d(mean, cvar, shift, B, N, S, eps, m * S, strips, counts, n, acq, cons=cn)
    k = w.k
    idx = torch.empty((B, k), dtype=torch.int64, device=dev)
    val = torch.empty((B, k), dtype=f32, device=dev)
    bt.boute_select_topk(acq, B, N, k, idx, val)
    torch.cuda.synchronize()
    st = bt.boute_gp_status(gp)
    gp.free()
    h = lambda a: a.cpu().numpy()
    return dict(status=st, Yin=h(Yin), mean=h(mean), cvar=h(cvar), shift=h(shift), pm=h(pm),
                pv=h(pv), strips=h(strips), counts=h(counts), acq=h(acq), idx=h(idx))


def _front_from_strips(strips, count):
    """Front points (f1, f2) of one draw from its strips 1 .. count-1."""
    return np.array([(strips[j, 0], strips[j, 2]) for j in range(1, count)], np.float64)


def _nehvi(fp, Yin, mean, cvar, shift, eps, cons):
    """The oracle acquisition on given intermediates (fp64 copies)."""
    return oracle.nehvi_mc(np.asarray(Yin, np.float64), np.asarray(mean, np.float64),
                           np.asarray(cvar, np.float64), np.asarray(shift, np.float64), eps,
                           fp.ref, cons=cons)


def _sensitivity(fp, dr, eps, cons, s2):
    """First-order change of the oracle acquisition when the posterior's
    outputs (mean and shifts, conditional variance, in-sample draws) move by
    their tolerance, objective by objective."""
    base = _nehvi(fp, dr.Yin, dr.mean, dr.cvar, dr.shift, eps, cons)
    tot = np.zeros_like(base)
    for t in range(dr.mean.shape[1]):
        s = np.sqrt(s2[t])
        dm = POST_REL * np.maximum(np.abs(dr.mean[:, t]), s)
        for sign in (1.0, -1.0):
            mm = dr.mean.copy()
            mm[:, t] += sign * dm
            dmean = np.abs(_nehvi(fp, dr.Yin, mm, dr.cvar, dr.shift, eps, cons) - base)
            vv = dr.cvar.copy()
            vv[:, t] = np.maximum(vv[:, t] + sign * POST_REL * s2[t], 0.0)
            dvar = np.abs(_nehvi(fp, dr.Yin, dr.mean, vv, dr.shift, eps, cons) - base)
            yy = dr.Yin.copy()
            yy[:, :, t] += sign * POST_REL * s
            dyin = np.abs(_nehvi(fp, yy, dr.mean, dr.cvar, dr.shift, eps, cons) - base)
            tot = np.maximum(tot, 2 * dmean + dvar + dyin)  # the shift moves like the mean
    return base, tot


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"w{c[0]}-N{c[1]}-n{c[2]}-S{c[3]}-B{c[4]}"
                         + ("-cons" if c[5] else ""))
def test_noisy_acquisition_matches_oracle(case):
    wi, N, n, S, B, constrained = case
    w = _workload(wi, N, n, S, B)
    hp = host_problem(w)
    z = np.stack([wl.insample_normals(w, b) for b in range(B)])  # B x m x S x n
    cons = _cons(hp) if constrained else None
    g = _gpu(hp, z, cons)
    assert g["status"] == 0
    for b in range(B):
        fp = oracle_fit(hp, b)
        s2 = hp.s2[b]
        dr = opl.noisy_draws(fp, hp.Xc[b], z[b])
        cb = None if cons is None else cons[b]
        # in-sample draws (S x n x m) and the joint posterior
        yin_g = np.transpose(g["Yin"][b], (1, 2, 0))
        err = np.abs(yin_g - dr.Yin) / np.sqrt(s2)[None, None, :]
        assert err.max() <= POST_REL, f"Yin err {err.max():.3g}"
        for t in range(w.m):
            check_mean(g["mean"][b, t], dr.mean[:, t], s2[t])
            ev = np.abs(g["cvar"][b, t] - np.maximum(dr.cvar[:, t], 0)) / s2[t]
            assert ev.max() <= POST_REL, f"cvar err {ev.max():.3g}"
            es = np.abs(g["shift"][b, t].T - dr.shift[:, t, :]) / np.sqrt(s2[t])
            assert es.max() <= POST_REL, f"shift err {es.max():.3g}"
        # the plain posterior on the same handle
        mean_o, var_o = opl.posterior(fp, hp.Xc[b])
        for t in range(w.m):
            check_mean(g["pm"][b, t], mean_o[:, t], s2[t])
            assert (np.abs(g["pv"][b, t] - var_o[:, t]) / s2[t]).max() <= POST_REL
        # fronts: bit-exact against the oracle's front of the GPU's draws, with
        # the reference point and thresholds rounded to fp32 as the kernel does
        ref32 = fp.ref.astype(np.float32).astype(np.float64)
        c32 = None if cb is None else np.asarray(cb, np.float32).astype(np.float64)
        for s in range(S):
            pts = yin_g[s].astype(np.float64)
            if c32 is not None:
                pts = pts[(pts <= c32).all(1)]
            mask, order = oracle.pareto_front(pts, ref32)
            want = pts[order][np.argsort(pts[order][:, 0], kind="stable")]
            got = _front_from_strips(g["strips"][b, s], int(g["counts"][b, s]))
            assert got.shape == want.shape and np.array_equal(got, want), f"front of draw {s}"
            st = g["strips"][b, s]
            assert st[0, 0] == -np.inf and st[0, 2] == np.float32(fp.ref[1])
        # the acquisition kernel on the GPU's intermediates
        a_at_g = _nehvi(fp, yin_g, g["mean"][b].T, g["cvar"][b].T,
                        np.transpose(g["shift"][b], (2, 0, 1)), hp.eps[b], c32)
        check_acq(g["acq"][b], a_at_g)
        # the whole chain against the oracle's own, and the selection
        o, sens = _sensitivity(fp, dr, hp.eps[b], cb, s2)
        tol = ACQ_REL * np.maximum(np.abs(o), ACQ_FLOOR * np.abs(o).max()) + 2 * sens
        e2e = np.abs(g["acq"][b] - o)
        assert np.all(e2e <= tol), f"acq e2e err {e2e.max():.3g} > tol at {np.argmax(e2e - tol)}"
        assert o.max() > 0
        check_topk_consistent_tol(g["idx"][b], o, w.k, tol)


def test_composite_kernel_noisy_draws():
    """The in-sample preparation reads the fit's factor, whatever the kernel."""
    w = _workload(1, 1024 + 9, 96, 48, 1, comp=True)
    hp = host_problem(w)
    z = np.stack([wl.insample_normals(w, 0)])
    g = _gpu(hp, z, None)
    assert g["status"] == 0
    fp = oracle_fit(hp, 0)
    dr = opl.noisy_draws(fp, hp.Xc[0], z[0])
    s2 = hp.s2[0]
    yin_g = np.transpose(g["Yin"][0], (1, 2, 0))
    assert (np.abs(yin_g - dr.Yin) / np.sqrt(s2)).max() <= POST_REL
    for t in range(w.m):
        check_mean(g["mean"][0, t], dr.mean[:, t], s2[t])
        assert (np.abs(g["cvar"][0, t] - np.maximum(dr.cvar[:, t], 0)) / s2[t]).max() <= POST_REL
        assert (np.abs(g["shift"][0, t].T - dr.shift[:, t, :]) / np.sqrt(s2[t])).max() <= POST_REL


def test_insample_limits():
    from paper_2602_10729_gb300 import boute as bt
    gp = bt.boute_gp_create(1, 129, 4, 2)
    with pytest.raises(bt.BouteError) as ei:
        bt.boute_gp_set_insample(gp, 16)
    assert ei.value.code == bt.BOUTE_ERR_UNSUPPORTED
    gp.free()
    gp = bt.boute_gp_create(1, 64, 4, 2)
    with pytest.raises(bt.BouteError):
        bt.boute_gp_set_insample(gp, 1025)
    bt.boute_gp_set_insample(gp, 16)
    with pytest.raises(bt.BouteError) as ei:
        bt.boute_gp_set_precision(gp, bt.BOUTE_PREC_FP64)
    assert ei.value.code == bt.BOUTE_ERR_UNSUPPORTED
    bt.boute_gp_set_insample(gp, 0)
    gp.free()


INSAMPLE_KEY = 0x6a09e667f3bcc909  # the engine's in-sample normals: seed ^ this key


def _engine_inputs(hp):
    import torch
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), device="cuda", dtype=dt)
    f64, f32 = torch.float64, torch.float32
    return (t(hp.X, f64), t(hp.Y, f64), t(hp.ls, f64), t(hp.s2, f64), t(hp.noise, f64),
            t(hp.ref, f64), t(hp.Xc, f32), t(hp.eps, f32))


def _engine_step(e, w, inputs, how="device"):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    if how == "host":
        hin = tuple(a.cpu().pin_memory() for a in inputs)
        idx = torch.empty((w.B, w.k), dtype=torch.int64).pin_memory()
        val = torch.empty((w.B, w.k), dtype=torch.float32).pin_memory()
        bt.boute_engine_step_host(e, *hin, idx, val)
        return idx.numpy().copy(), val.numpy().copy()
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device="cuda")
    val = torch.empty((w.B, w.k), dtype=torch.float32, device="cuda")
    if how == "legacy":
        torch.cuda.synchronize()
        bt.boute_engine_step(e, *inputs, idx, val, stream=0)
    else:
        bt.boute_engine_step(e, *inputs, idx, val)
    return idx.cpu().numpy(), val.cpu().numpy()


@pytest.mark.parametrize("case", [(1, 3000 + 77, 128, 128, 1, False, 7),
                                  (4, 999, 64, 64, 2, True, 0)],
                         ids=["medium-n128-S128", "batched-n64-S64-cons"])
def test_engine_noisy_step_matches_oracle(case):
    """The whole noisy step through the engine: graph replay, host inputs and
    eager launches agree value for value, and the selection is the oracle's
    (in-sample normals regenerated from the documented key)."""
    import torch

    from paper_2602_10729_gb300 import boute as bt
    wi, N, n, S, B, constrained, seed = case
    w = _workload(wi, N, n, S, B)
    hp = host_problem(w)
    cons = _cons(hp) if constrained else None
    e = bt.Engine(B, n, w.d, w.m, N, bt.BOUTE_ACQ_NEHVI, S, w.k)
    if seed:
        bt.boute_engine_set_normals(e, seed)
    if cons is not None:
        bt.boute_engine_set_constraints(e, torch.as_tensor(cons, dtype=torch.float64))
    inputs = _engine_inputs(hp)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        ref_idx, ref_val = _engine_step(e, w, inputs)
        for how in ("device", "host", "legacy"):
            idx, val = _engine_step(e, w, inputs, how)
            assert np.array_equal(idx, ref_idx), how
            assert np.array_equal(val, ref_val), how
    e.free()
    z = oracle.base_normals(seed ^ INSAMPLE_KEY, B, w.m * S, 1, n).reshape(B, w.m, S, n)
    for b in range(B):
        fp = oracle_fit(hp, b)
        dr = opl.noisy_draws(fp, hp.Xc[b], z[b])
        cb = None if cons is None else cons[b]
        o, sens = _sensitivity(fp, dr, hp.eps[b], cb, hp.s2[b])
        tol = ACQ_REL * np.maximum(np.abs(o), ACQ_FLOOR * np.abs(o).max()) + 2 * sens
        check_topk_consistent_tol(ref_idx[b], o, w.k, tol)
        np.testing.assert_allclose(ref_val[b], o[ref_idx[b]], rtol=0, atol=float(tol.max()))


def test_engine_noisy_set_n_matches_fresh_engine():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    base = _workload(1, 1024 + 3, 128, 64, 1)
    e = bt.Engine(1, 128, base.d, 2, base.N, bt.BOUTE_ACQ_NEHVI, 64, base.k)
    bt.boute_engine_set_normals(e, 5)
    stream = torch.cuda.Stream()
    for n in (128, 57, 100):
        w = _workload(1, 1024 + 3, n, 64, 1)
        hp = host_problem(w)
        inputs = _engine_inputs(hp)
        bt.boute_engine_set_n(e, n)
        fresh = bt.Engine(1, n, w.d, 2, w.N, bt.BOUTE_ACQ_NEHVI, 64, w.k)
        bt.boute_engine_set_normals(fresh, 5)
        with torch.cuda.stream(stream):
            ri, rv = _engine_step(fresh, w, inputs)
            for how in ("device", "device", "legacy"):
                idx, val = _engine_step(e, w, inputs, how)
                assert np.array_equal(idx, ri) and np.array_equal(val, rv), (n, how)
        fresh.free()
    e.free()

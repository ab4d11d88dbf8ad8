"""Optimising the acquisition over the decision space (Sec. 5.2 step (ii))
on the GPU against the oracle: the sample-average MC acquisition and its
gradient at given points (steps = 0), and projected Adam ascent from the
best candidates of a pool (the end values against the oracle's optimiser,
which takes the same steps in fp64; the GPU's reported values re-evaluated
by the oracle at the GPU's end points)."""
import numpy as np
import pytest

from _pipeline import host_problem, oracle_fit
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _setup(hp, S, seed=3):
    """The GPU fit and the front's strips of problem set hp; shared normals."""
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = hp.w
    B, n, d, m = w.B, w.n, w.d, w.m
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), device="cuda", dtype=dt)
    f64, f32 = torch.float64, torch.float32
    X, Y = t(hp.X, f64), t(hp.Y, f64)
    Ys = torch.empty_like(Y)
    bt.boute_standardize(Y, Ys)
    gp = bt.boute_gp_create(B, n, d, m)
    bt.boute_gp_fit(gp, X, Ys, t(hp.ls, f64), t(hp.s2, f64), t(hp.noise, f64))
    assert bt.boute_gp_status(gp) == 0
    ref = t(hp.ref, f64)
    mask = torch.empty((B, n), dtype=torch.uint8, device="cuda")
    front = torch.zeros((B, n, m), dtype=f64, device="cuda")
    P = torch.empty(B, dtype=torch.int32, device="cuda")
    bt.boute_pareto_front(Ys, B, n, m, ref, mask, front, P)
    cap = 2 * n + 2
    lower = torch.empty((B, cap, m), dtype=f32, device="cuda")
    upper = torch.empty_like(lower)
    K = torch.empty(B, dtype=torch.int32, device="cuda")
    bt.boute_box_decompose(front, P, B, n, m, ref, lower, upper, K)
    eps = np.random.default_rng(seed).standard_normal((2, S)).astype(np.float32)
    return gp, lower, upper, K, cap, t(eps, f32), eps.astype(np.float64)


def _run(gp, strips, epsd, X0, steps, lr, d):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    lower, upper, K, cap = strips
    B, P = X0.shape[0], X0.shape[1]
    x0 = torch.as_tensor(np.ascontiguousarray(X0, np.float32), device="cuda")
    X = torch.empty_like(x0)
    acq = torch.empty((B, P), dtype=torch.float32, device="cuda")
    grad = torch.empty_like(x0)
    lo = torch.zeros(d, dtype=torch.float32, device="cuda")
    hi = torch.ones(d, dtype=torch.float32, device="cuda")
    bt.boute_acq_optimize(gp, lower, upper, K, cap, epsd, epsd.shape[1], x0, P, lo, hi, steps, lr,
                          X, acq, grad)
    torch.cuda.synchronize()
    return X.cpu().numpy(), acq.cpu().numpy(), grad.cpu().numpy()


@pytest.mark.parametrize("wi,n,S,B", [(2, 96, 64, 1), (1, 128, 128, 1), (4, 40, 32, 2)])
def test_value_and_gradient_match_oracle(wi, n, S, B):
    w = wl.scaled(wl.WORKLOADS[wi], N=64, B=B, n=n)
    hp = host_problem(w)
    gp, lower, upper, K, cap, epsd, eps = _setup(hp, S)
    rng = np.random.default_rng(11)
    X0 = rng.uniform(0.05, 0.95, (B, 24, w.d)).astype(np.float32)
    X, acq, grad = _run(gp, (lower, upper, K, cap), epsd, X0, 0, 0.01, w.d)
    gp.free()
    assert np.array_equal(X, X0)
    for b in range(B):
        fp = oracle_fit(hp, b)
        vals, grads = zip(*(opl.mc_hvi_value_grad(fp, X0[b, p].astype(np.float64), eps)
                            for p in range(X0.shape[1])))
        vals, grads = np.array(vals), np.array(grads)
        scale = np.abs(vals).max()
        assert scale > 0
        np.testing.assert_allclose(acq[b], vals, rtol=1e-4, atol=1e-6 * scale)
        gs = np.abs(grads).max()
        np.testing.assert_allclose(grad[b], grads, rtol=1e-3, atol=2e-4 * gs)


@pytest.mark.parametrize("wi,n,S", [(2, 96, 64), (1, 64, 64)])
def test_ascent_from_the_pool_best_matches_oracle(wi, n, S):
    w = wl.scaled(wl.WORKLOADS[wi], N=2048, B=1, n=n)
    hp = host_problem(w)
    gp, lower, upper, K, cap, epsd, eps = _setup(hp, S, seed=5)
    fp = oracle_fit(hp, 0)
    # starting points: the pool's best by the same acquisition
    pool = hp.Xc[0].astype(np.float64)
    pv = np.array([opl.mc_hvi_value_grad(fp, x, eps)[0] for x in pool[:512]])
    starts = pool[np.argsort(-pv)[:6]].astype(np.float32)
    steps, lr = 40, 0.01
    X, acq, _ = _run(gp, (lower, upper, K, cap), epsd, starts[None], steps, lr, w.d)
    gp.free()
    Xo, ao = opl.optimize_acq(fp, starts.astype(np.float64), eps, np.zeros(w.d), np.ones(w.d),
                              steps, lr)
    a0 = np.array([opl.mc_hvi_value_grad(fp, s.astype(np.float64), eps)[0] for s in starts])
    ag = np.array([opl.mc_hvi_value_grad(fp, x.astype(np.float64), eps)[0] for x in X[0]])
    scale = np.abs(ao).max()
    assert (X[0] >= 0).all() and (X[0] <= 1).all()
    np.testing.assert_allclose(acq[0], ag, rtol=1e-4, atol=1e-6 * scale)  # the reported values
    assert (ag >= a0 - 1e-5 * scale).all()  # ascent from every start
    np.testing.assert_allclose(ag, ao, rtol=0, atol=1e-3 * scale)  # the oracle's end values
    assert ao.max() > a0.max()  # the steps improve on the pool's best


def test_unsupported_requests():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = wl.scaled(wl.WORKLOADS[3], N=64, B=1, n=32)  # three objectives
    hp = host_problem(w)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), device="cuda", dtype=dt)
    gp = bt.boute_gp_create(1, w.n, w.d, 3)
    z = torch.zeros((1, 4, w.d), device="cuda")
    a = torch.zeros((1, 4), device="cuda")
    box = torch.zeros((1, 66, 3), device="cuda")
    K = torch.zeros(1, dtype=torch.int32, device="cuda")
    e = torch.zeros((2, 8), device="cuda")
    lo = torch.zeros(w.d, device="cuda")
    with pytest.raises(bt.BouteError) as ei:
        bt.boute_acq_optimize(gp, box, box, K, 66, e, 8, z, 4, lo, lo + 1, 1, 0.01, z, a)
    assert ei.value.code == bt.BOUTE_ERR_UNSUPPORTED
    with pytest.raises(bt.BouteError) as ei:
        bt.boute_acq_optimize(gp, box, box, K, 66, e, 8, z, 4, lo, lo + 1, 1, 0.0, z, a)
    assert ei.value.code == bt.BOUTE_ERR_INVALID_ARG
    gp.free()
    del hp, t

"""The FP64 tier of the posterior (Sec. 6 and Appendix C: the paper runs its
GP in double precision) against the fp64 oracle at 1e-10: the mean relative
to max(|mean|, s), the variance relative to the prior variance s2, on the
tiny and medium workloads' shapes and on a problem with per-objective
hyperparameters; and the requests the tier does not serve."""
import numpy as np
import pytest

from _pipeline import host_problem
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

FP64_REL = 1e-10


def _fp64_posterior(hp, N=None):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = hp.w
    B, n, d, m = w.B, w.n, w.d, w.m
    N = hp.Xc.shape[1] if N is None else N
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a), dtype=dt, device="cuda")
    Y = t(hp.Y, torch.float64)
    Ys = torch.empty_like(Y)
    bt.boute_standardize(Y, Ys)
    gp = bt.boute_gp_create(B, n, d, m)
    bt.boute_gp_set_precision(gp, bt.BOUTE_PREC_FP64)
    bt.boute_gp_fit(gp, t(hp.X, torch.float64), Ys, t(hp.ls, torch.float64),
                    t(hp.s2, torch.float64), t(hp.noise, torch.float64))
    st = bt.boute_gp_status(gp)
    mean = torch.empty((B, m, N), dtype=torch.float64, device="cuda")
    var = torch.empty_like(mean)
    if st == 0:
        bt.boute_gp_posterior_fp64(gp, t(hp.Xc[:, :N], torch.float32), N, mean, var)
        torch.cuda.synchronize()
    gp.free()
    return st, mean.cpu().numpy(), var.cpu().numpy()


def _check(hp, N=None):
    st, mean, var = _fp64_posterior(hp, N)
    assert st == 0
    for b in range(hp.w.B):
        fp = opl.fit_problem(hp.X[b], hp.Y[b], hp.ls[b], hp.s2[b], hp.noise[b], hp.ref[b])
        mo, vo = opl.posterior(fp, hp.Xc[b, :mean.shape[2]])
        for t in range(hp.w.m):
            s = np.sqrt(fp.s2[t])
            em = np.abs(mean[b, t] - mo[:, t]) / np.maximum(np.abs(mo[:, t]), s)
            ev = np.abs(var[b, t] - vo[:, t]) / fp.s2[t]
            assert em.max() <= FP64_REL, f"mean rel err {em.max():.3g}"
            assert ev.max() <= FP64_REL, f"var rel err {ev.max():.3g}"
            assert np.all(var[b, t] >= 0)


@pytest.mark.parametrize("wi,N", [(0, 4096), (1, 6000)])
def test_fp64_tier_matches_oracle_on_workloads(wi, N):
    _check(host_problem(wl.scaled(wl.WORKLOADS[wi], N=N)))


def test_fp64_tier_per_objective_hyperparameters():
    from test_gpu_edge import rand_problem
    rng = np.random.default_rng(8)
    hp = rand_problem(9, 70, 5, 2, 333)
    hp.ls[0] = rng.uniform(0.2, 0.6, (2, 5))
    hp.s2[0] = [0.5, 2.5]
    hp.noise[0] = [1e-3, 1e-4]
    _check(hp)


def test_fp64_tier_requests_it_does_not_serve():
    from paper_2602_10729_gb300 import boute as bt
    gp = bt.boute_gp_create(1, 129, 3, 1)  # n beyond 128
    with pytest.raises(bt.BouteError) as e:
        bt.boute_gp_set_precision(gp, bt.BOUTE_PREC_FP64)
    assert e.value.code == bt.BOUTE_ERR_UNSUPPORTED
    gp.free()
    gp = bt.boute_gp_create(1, 16, 4, 1)
    import torch
    with pytest.raises(bt.BouteError) as e:  # not switched to fp64
        bt.boute_gp_posterior_fp64(gp, torch.zeros((1, 4, 4), device="cuda"), 4,
                                   torch.zeros((1, 1, 4), dtype=torch.float64, device="cuda"),
                                   torch.zeros((1, 1, 4), dtype=torch.float64, device="cuda"))
    assert e.value.code == bt.BOUTE_ERR_INVALID_ARG
    bt.boute_gp_set_kernel(gp, 2, np.array([[[0.5, 0.1, 0.05, 0.3, 0.7]]]))  # composite
    with pytest.raises(bt.BouteError) as e:
        bt.boute_gp_set_precision(gp, bt.BOUTE_PREC_FP64)
    assert e.value.code == bt.BOUTE_ERR_UNSUPPORTED
    gp.free()


def test_fp64_tier_reports_a_singular_kernel_matrix():
    from test_gpu_edge import custom
    from paper_2602_10729_gb300 import boute as bt
    X = np.array([[0.1, 0.2], [0.1, 0.2], [0.5, 0.5], [0.7, 0.1]])
    Y = np.array([[0.0, 1.0], [0.0, 1.0], [1.0, 0.0], [0.5, 0.5]])
    st, _, _ = _fp64_posterior(custom(X, Y, np.zeros((10, 2)), noise=0.0))
    assert st == bt.BOUTE_ERR_NOT_PD

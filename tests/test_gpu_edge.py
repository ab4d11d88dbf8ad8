"""Edge cases of the CUDA path against the oracle: ragged and tiny sizes, one
training point, several output-column passes, extreme dimensions, an empty
front, candidates on training points, zero variance, ties in selection,
shared base normals, per-objective hyperparameters, a singular kernel matrix
and invalid arguments."""
import numpy as np
import pytest

import oracle
from _pipeline import (HostProblem, check_acq, check_acq_end_to_end, check_mean, check_var,
                       gpu_pipeline, host_problem, oracle_fit)
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def custom(X, Y, Xc, *, ls=None, s2=None, noise=None, ref=None, mode="ehvi", S=0, k=4,
           eps=None):
    X = np.asarray(X, np.float64)[None] if np.ndim(X) == 2 else np.asarray(X, np.float64)
    Y = np.asarray(Y, np.float64)[None] if np.ndim(Y) == 2 else np.asarray(Y, np.float64)
    Xc = np.asarray(Xc, np.float32)[None] if np.ndim(Xc) == 2 else np.asarray(Xc, np.float32)
    B, n, d = X.shape
    m = Y.shape[2]
    N = Xc.shape[1]
    ls = np.full((B, m, d), 0.3) if ls is None else np.broadcast_to(ls, (B, m, d)).copy()
    s2 = np.ones((B, m)) if s2 is None else np.broadcast_to(s2, (B, m)).copy()
    noise = np.full((B, m), 1e-4) if noise is None else np.broadcast_to(noise, (B, m)).copy()
    ref = np.full((B, m), 1.1) if ref is None else np.broadcast_to(ref, (B, m)).copy()
    w = wl.Workload("custom", B, n, d, m, N, mode, S, min(k, N), tuple(range(B)), 0,
                    ref=tuple(ref[0]))
    return HostProblem(w, X, Y, ls, s2, noise, ref, Xc, eps)


def compare(hp, check_topk=True):
    g = gpu_pipeline(hp)
    assert g["status"] == 0, g["status"]
    w = hp.w
    for b in range(w.B):
        fp = opl.fit_problem(hp.X[b], hp.Y[b], hp.ls[b], hp.s2[b], hp.noise[b], hp.ref[b])
        assert g["mask"][b].tolist() == fp.mask.tolist()
        assert int(g["P"][b]) == fp.front.shape[0]
        mean, var = opl.posterior(fp, hp.Xc[b])
        for t in range(w.m):
            check_mean(g["mean"][b, t], mean[:, t], fp.s2[t])
            check_var(g["var"][b, t], var[:, t], fp.s2[t])
        eps = None if hp.eps is None else hp.eps[b]
        check_acq_end_to_end(g["acq"][b], lambda mm, vv: opl.acquisition(fp, mm, vv, w.mode, eps),
                             g["mean"][b].T, g["var"][b].T, mean, var, fp.s2)
    return g


def rand_problem(seed, n, d, m, N, mode="ehvi", S=0, **kw):
    rng = np.random.default_rng(seed)
    X = rng.random((n, d))
    Y = np.stack([((X - c) ** 2).sum(1) for c in np.linspace(0.2, 0.8, m)], 1)
    Y += rng.normal(0, 0.01, Y.shape)
    Xc = rng.random((N, d)).astype(np.float32)
    eps = rng.standard_normal((1, N, m, S)).astype(np.float32) if mode == "mc" else None
    return custom(X, Y, Xc, mode=mode, S=S, eps=eps, **kw)


@pytest.mark.parametrize("N", [1, 2, 127, 128, 129, 300])
def test_ragged_candidate_counts(N):
    compare(rand_problem(1, 20, 4, 2, N))


@pytest.mark.parametrize("n", [1, 2, 31, 33, 97, 129, 150, 160, 161, 255, 257, 600])
def test_training_set_sizes_and_column_passes(n):
    compare(rand_problem(2, n, 5, 2, 400))


@pytest.mark.parametrize("d", [1, 3, 8, 9, 13, 17, 25, 32])
def test_dimensions(d):
    # lengthscale 0.2 sqrt(d) as in the workloads; 1-D with few points keeps
    # the kernel matrix well conditioned (see the ill-conditioned test below)
    n, ls = (6, 0.1) if d == 1 else (40, 0.2 * np.sqrt(d))
    compare(rand_problem(3, n, d, 2, 300, ls=ls))


@pytest.mark.parametrize("n,d,m,N,mode,S", [(600, 20, 2, 700, "ehvi", 0),
                                            (777, 24, 3, 385, "mc", 64),
                                            (97, 32, 3, 257, "mc", 64)])
def test_wide_candidates_large_and_ragged(n, d, m, N, mode, S):
    # d > 16: the builders take candidate rows in pairs; n > 512 adds the
    # cached K* chunks of a second group; n, N not multiples of the chunk and
    # the tile; n = 777 with three objectives puts the MC kernel's boxes
    # (2n + 2) just under 48 KB of dynamic shared memory, beside its static
    # staging
    compare(rand_problem(13, n, d, m, N, mode=mode, S=S, ls=0.2 * np.sqrt(d)))


@pytest.mark.parametrize("n", [420, 440])
def test_kstar_side_input_near_48kb(n):
    # K* beside the fit (the engine, few candidates): the side input of
    # n = 420 .. 448 points at d = 12 needs just under 48 KB of dynamic shared
    # memory next to the K* kernel's static array
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = wl.scaled(wl.WORKLOADS[1], N=2048 + 5, B=1, n=n)
    hp = host_problem(w)
    dev = torch.device("cuda")
    t = lambda a, dt: torch.as_tensor(a, dtype=dt, device=dev)
    e = bt.Engine(1, w.n, w.d, w.m, w.N, bt.BOUTE_ACQ_MC_HVI, w.S, w.k)
    idx = torch.empty((1, w.k), dtype=torch.int64, device=dev)
    val = torch.empty((1, w.k), dtype=torch.float32, device=dev)
    bt.boute_engine_step(e, t(hp.X, torch.float64), t(hp.Y, torch.float64),
                         t(hp.ls, torch.float64), t(hp.s2, torch.float64),
                         t(hp.noise, torch.float64), t(hp.ref, torch.float64),
                         t(hp.Xc, torch.float32), t(hp.eps, torch.float32), idx, val)
    mean = torch.empty((1, w.m, w.N), dtype=torch.float32, device=dev)
    var = torch.empty_like(mean)
    bt.boute_engine_scores(e, None, mean, var)
    torch.cuda.synchronize()
    e.free()
    fp = oracle_fit(hp, 0)
    mo, vo = opl.posterior(fp, hp.Xc[0])
    for tt in range(w.m):
        check_mean(mean[0, tt].cpu().numpy(), mo[:, tt], fp.s2[tt])
        check_var(var[0, tt].cpu().numpy(), vo[:, tt], fp.s2[tt])


def test_ill_conditioned_problem_meets_fp32_error_bound():
    """40 points on a line with lengthscale 0.3: cond(K) ~ 2e5, |alpha| ~ 1e3.
    The mean meets 1e-5 (its ill-conditioned rows take the fp64 path); the
    variance s2 - ||L^-1 k*||^2 must stay within the error bound of an
    fp32-accurate contraction, eps32 * s2 times cond-scaled terms."""
    hp = rand_problem(12, 40, 1, 2, 300)
    g = gpu_pipeline(hp)
    assert g["status"] == 0
    fp = opl.fit_problem(hp.X[0], hp.Y[0], hp.ls[0], hp.s2[0], hp.noise[0], hp.ref[0])
    mean, var = opl.posterior(fp, hp.Xc[0])
    eps32 = np.finfo(np.float32).eps
    for t in range(2):
        Ks = np.array([[oracle.matern52(c.astype(np.float64), x, hp.ls[0][t], hp.s2[0][t])
                        for x in hp.X[0]] for c in hp.Xc[0]])
        check_mean(g["mean"][0, t], mean[:, t], fp.s2[t])
        W = np.linalg.inv(fp.L[t])
        v = Ks @ W.T
        bound_v = 64 * eps32 * 2 * (np.abs(v) * (np.abs(Ks) @ np.abs(W.T))).sum(1) + 1e-5
        assert np.all(np.abs(g["var"][0, t] - var[:, t]) <= bound_v)


def test_three_objectives_monte_carlo_and_box_decomposition():
    hp = rand_problem(4, 90, 6, 3, 500, mode="mc", S=64)
    g = compare(hp)
    # the boxes tile the improvement region: their volume inside [lb, ref]
    # equals vol([lb, ref]) - HV(front)
    fp = opl.fit_problem(hp.X[0], hp.Y[0], hp.ls[0], hp.s2[0], hp.noise[0], hp.ref[0])
    K = int(g["K"][0])
    lo, up = g["lower"][0][:K].astype(np.float64), g["upper"][0][:K].astype(np.float64)
    lb = fp.front.min(0) - 1.0 if len(fp.front) else hp.ref[0] - 1.0
    vol = np.prod(np.clip(up - np.maximum(lo, lb), 0, None), 1).sum()
    want = np.prod(hp.ref[0] - lb) - oracle.hv(fp.front, hp.ref[0])
    assert vol == pytest.approx(want, rel=1e-5)
    assert K <= 2 * len(fp.front) + 1


def test_monte_carlo_scalar_path_and_shared_normals():
    # S = 50 is not a multiple of 128 (scalar path); also shared normals
    hp = rand_problem(5, 50, 4, 2, 260, mode="mc", S=50)
    compare(hp)
    import torch

    from paper_2602_10729_gb300 import boute as bt
    fp = opl.fit_problem(hp.X[0], hp.Y[0], hp.ls[0], hp.s2[0], hp.noise[0], hp.ref[0])
    mean, var = opl.posterior(fp, hp.Xc[0])
    eps1 = hp.eps[0, :1]  # one m x S block for every candidate
    want = oracle.mc_hvi(mean.astype(np.float32).astype(np.float64),
                         var.astype(np.float32).astype(np.float64), eps1, fp.front, fp.ref,
                         eps_stride=0)
    dev = "cuda"
    n, m, N = hp.w.n, 2, 260
    front = torch.zeros((1, n, m), dtype=torch.float64, device=dev)
    front[0, :len(fp.front)] = torch.as_tensor(fp.front)
    P = torch.tensor([len(fp.front)], dtype=torch.int32, device=dev)
    ref = torch.as_tensor(fp.ref[None], device=dev)
    cap = 2 * n + 2
    lower = torch.empty((1, cap, m), dtype=torch.float32, device=dev)
    upper = torch.empty_like(lower)
    K = torch.empty(1, dtype=torch.int32, device=dev)
    bt.boute_box_decompose(front, P, 1, n, m, ref, lower, upper, K)
    acq = torch.empty((1, N), dtype=torch.float32, device=dev)
    bt.boute_acq_mc_hvi(torch.as_tensor(mean.T.astype(np.float32)[None].copy(), device=dev),
                        torch.as_tensor(var.T.astype(np.float32)[None].copy(), device=dev), 1, N,
                        m, lower, upper, K, cap, torch.as_tensor(eps1, device=dev), hp.w.S, 0, acq)
    check_acq(acq.cpu().numpy()[0], want)


def test_empty_front():
    hp = rand_problem(6, 30, 3, 2, 200, ref=-5.0)  # nothing is better than ref
    g = compare(hp)
    assert int(g["P"][0]) == 0


def test_candidates_on_training_points():
    rng = np.random.default_rng(7)
    X = rng.random((25, 3)).astype(np.float32).astype(np.float64)
    Y = np.stack([X.sum(1), (1 - X).sum(1)], 1) + rng.normal(0, 0.01, (25, 2))
    hp = custom(X, Y, X.astype(np.float32), noise=1e-6)
    g = compare(hp)
    assert g["var"].max() < 1e-3


def test_per_objective_hyperparameters():
    """Per-objective lengthscales over an order of magnitude and noise down to
    1e-5: sum_j |K*_j alpha_j| reaches about 220 times the mean's scale, and
    the mean must still meet 1e-5 (the fp32 K* with its exponent-rounding
    correction and compensated sums)."""
    rng = np.random.default_rng(8)
    hp = rand_problem(9, 70, 5, 2, 333)
    hp.ls[0] = rng.uniform(0.1, 1.5, (2, 5))
    hp.s2[0] = [0.5, 2.5]
    hp.noise[0] = [1e-3, 1e-5]
    compare(hp)


@pytest.mark.parametrize("ls_range,noise", [((0.3, 1.5), (1e-3, 1e-4)), ((0.5, 2.0), (1e-3, 1e-5)),
                                            ((0.1, 1.5), (1e-5, 1e-6))])
def test_ill_conditioned_means(ls_range, noise):
    """Longer lengthscales or smaller noise: sum_j |K*_j alpha_j| reaches 270
    to 590 times the mean's scale. Rows beyond 256 times take the fp64 path;
    mean and variance meet 1e-5 everywhere."""
    rng = np.random.default_rng(8)
    hp = rand_problem(9, 70, 5, 2, 333)
    hp.ls[0] = rng.uniform(*ls_range, (2, 5))
    hp.s2[0] = [0.5, 2.5]
    hp.noise[0] = list(noise)
    g = gpu_pipeline(hp)
    assert g["status"] == 0
    fp = opl.fit_problem(hp.X[0], hp.Y[0], hp.ls[0], hp.s2[0], hp.noise[0], hp.ref[0])
    mean, var = opl.posterior(fp, hp.Xc[0])
    for t in range(2):
        check_mean(g["mean"][0, t], mean[:, t], fp.s2[t])
        check_var(g["var"][0, t], var[:, t], fp.s2[t])


def test_far_candidates_and_zero_variance_ehvi():
    hp = rand_problem(10, 30, 3, 2, 150)
    hp.Xc[0, :20] += 50.0  # far field: mean 0, var s2
    compare(hp)


# k <= 32 takes the warp-register path, larger k the segment sort; N spans one
# block, several, and more than 256 first-level blocks (larger blocks)
@pytest.mark.parametrize("N,k", [(5000, 40), (5000, 32), (5000, 1), (2048, 7), (40, 32),
                                 (700_001, 32), (700_001, 17), (70_000, 33)])
def test_topk_ties_nan_and_negative_zero(N, k):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    rng = np.random.default_rng(11)
    B = 3
    v = np.round(rng.random((B, N)), 2).astype(np.float32)
    v[0, [i for i in (3, 99) if i < N]] = np.nan
    v[1, :50] = -0.0
    v[1, 50:] = -1.0
    v[2, :] = 0.25  # all equal: the first k indices
    v[0, -1] = 2.0  # the maximum in the ragged tail
    a = torch.as_tensor(v, device="cuda")
    idx = torch.empty((B, k), dtype=torch.int64, device="cuda")
    val = torch.empty((B, k), dtype=torch.float32, device="cuda")
    bt.boute_select_topk(a, B, N, k, idx, val)
    for b in range(B):
        oi, ov = oracle.topk(v[b].astype(np.float64), k)
        assert idx[b].cpu().numpy().tolist() == oi.tolist()
    assert idx[2].cpu().numpy().tolist() == list(range(k))


def test_singular_kernel_matrix_reports_not_pd():
    X = np.array([[0.1, 0.2], [0.1, 0.2], [0.5, 0.5], [0.7, 0.1]])
    Y = np.array([[0.0, 1.0], [0.0, 1.0], [1.0, 0.0], [0.5, 0.5]])
    hp = custom(X, Y, np.zeros((10, 2)), noise=0.0)
    g = gpu_pipeline(hp)
    from paper_2602_10729_gb300 import boute as bt
    assert g["status"] == bt.BOUTE_ERR_NOT_PD
    with pytest.raises(oracle.NotPositiveDefinite):
        oracle.gp_fit(X, Y[:, 0], np.full(2, 0.3), 1.0, 0.0)


def test_invalid_arguments_raise():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    with pytest.raises(bt.BouteError) as e:
        bt.boute_gp_create(1, 10, 40, 2)
    assert e.value.code == bt.BOUTE_ERR_INVALID_ARG
    a = torch.zeros((1, 10), device="cuda")
    idx = torch.empty((1, 11), dtype=torch.int64, device="cuda")
    val = torch.empty((1, 11), device="cuda")
    with pytest.raises(bt.BouteError):
        bt.boute_select_topk(a, 1, 10, 11, idx, val)

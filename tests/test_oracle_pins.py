"""Pins of the CPU oracle against facts that do not come from the oracle itself:
closed forms, a different special-function route to the same kernel, library
linear algebra on the same definitions, brute-force enumeration, quadrature,
invariants and hand-derived worked examples (tests/golden/). A plausible
mistake anywhere in the oracle (dropped term, wrong sign or index, transposed
operand) fails at least one of these."""
import json
import math
import os

import numpy as np
import pytest
import scipy.integrate
import scipy.linalg
import scipy.special

import oracle
from oracle import pipeline
from paper_2602_10729_gb300 import workloads as wl

GOLD = os.path.join(os.path.dirname(__file__), "golden", "hypervolume_cases.json")


# --------------------------------------------------------------- Matern 5/2
def _matern_bessel(r, nu, s2):
    """General Matern covariance through the modified Bessel function K_nu."""
    if r == 0:
        return s2
    z = math.sqrt(2 * nu) * r
    return s2 * 2 ** (1 - nu) / scipy.special.gamma(nu) * z ** nu * scipy.special.kv(nu, z)


@pytest.mark.parametrize("r", [0.0, 1e-3, 0.1, 0.5, 1.0, 2.0, 3.7, 8.0])
def test_matern52_equals_general_matern_at_nu_2p5(r):
    ls = np.array([0.3, 1.7, 0.9])
    u = np.array([0.2, -0.5, 0.4])
    u = u / np.linalg.norm(u / ls) * r if r > 0 else np.zeros(3)  # scaled distance r
    a = np.array([0.1, 0.2, 0.3])
    got = oracle.matern52(a, a + u, ls, 1.7)
    assert got == pytest.approx(_matern_bessel(r, 2.5, 1.7), rel=1e-12, abs=1e-300)


def test_matern52_symmetry_and_ard():
    rng = np.random.default_rng(3)
    a, b = rng.random(5), rng.random(5)
    ls = rng.random(5) + 0.2
    assert oracle.matern52(a, b, ls) == oracle.matern52(b, a, ls)
    # a lengthscale of infinity removes that dimension from the distance
    ls2 = ls.copy(); ls2[2] = np.inf
    b2 = b.copy(); b2[2] = a[2]
    assert oracle.matern52(a, b, ls2) == pytest.approx(oracle.matern52(a, b2, ls), rel=1e-15)


# ------------------------------------------------------------ standardise
def test_standardize_moments_and_affine_invariance():
    rng = np.random.default_rng(0)
    Y = rng.normal(3.0, 2.0, (50, 3))
    Ys = oracle.standardize(Y)
    np.testing.assert_allclose(Ys.mean(0), 0, atol=1e-14)
    np.testing.assert_allclose(Ys.std(0, ddof=1), 1, rtol=1e-13)
    np.testing.assert_allclose(oracle.standardize(4.0 * Y - 7.0), Ys, atol=1e-13)
    # constant column / single row: divided by one
    Yc = np.ones((4, 1)) * 5.0
    np.testing.assert_allclose(oracle.standardize(Yc), 0.0)
    np.testing.assert_allclose(oracle.standardize(np.array([[2.0, 3.0]])), 0.0)


# --------------------------------------------------------------- GP fit
def _kernel_matrix(X, ls, s2, noise):
    n = len(X)
    K = np.array([[oracle.matern52(X[i], X[j], ls, s2) for j in range(n)] for i in range(n)])
    return K + noise * np.eye(n)


@pytest.mark.parametrize("wi", [0, 1, 4])
def test_cholesky_residual_and_library_factor(wi):
    w = wl.WORKLOADS[wi]
    X, Y = wl.training_set(w, 0)
    ls, s2, noise = wl.hyperparameters(w, 0)
    y = oracle.standardize(Y)[:, 0]
    L, alpha = oracle.gp_fit(X, y, ls[0], s2[0], noise[0])
    K = _kernel_matrix(X, ls[0], s2[0], noise[0])
    assert np.linalg.norm(L @ L.T - K) / np.linalg.norm(K) < 1e-12
    assert np.all(np.triu(L, 1) == 0) and np.all(np.diag(L) > 0)
    np.testing.assert_allclose(L, scipy.linalg.cholesky(K, lower=True), atol=1e-12)
    np.testing.assert_allclose(alpha, np.linalg.solve(K, y), rtol=1e-9, atol=1e-10)


def test_cholesky_tiny_matches_gauss_jordan_solve():
    X = np.array([[0.0, 0.0], [0.3, 0.1], [0.9, 0.5]])
    ls = np.array([0.5, 0.7])
    y = np.array([1.0, -2.0, 0.5])
    L, alpha = oracle.gp_fit(X, y, ls, 2.0, 0.01)
    K = _kernel_matrix(X, ls, 2.0, 0.01)
    # Gauss-Jordan elimination on [K | y], written out
    A = np.hstack([K, y[:, None]])
    for c in range(3):
        A[c] /= A[c, c]
        for r in range(3):
            if r != c:
                A[r] -= A[r, c] * A[c]
    np.testing.assert_allclose(alpha, A[:, 3], rtol=1e-12)


def test_not_positive_definite_is_reported():
    X = np.array([[0.1, 0.2], [0.1, 0.2], [0.5, 0.5]])  # duplicate rows, no noise
    with pytest.raises(oracle.NotPositiveDefinite):
        oracle.gp_fit(X, np.zeros(3), np.ones(2), 1.0, 0.0)


# ------------------------------------------------------------ posterior
def _fit(X, y, ls, s2, noise):
    L, a = oracle.gp_fit(X, y, ls, s2, noise)
    return L, a


def test_posterior_matches_schur_complement_by_library_solve():
    w = wl.WORKLOADS[0]
    X, Y = wl.training_set(w, 0)
    ls, s2, noise = wl.hyperparameters(w, 0)
    y = oracle.standardize(Y)[:, 1]
    L, a = _fit(X, y, ls[1], s2[1], noise[1])
    Xc = wl.candidates(w, 0, 0, 64)
    mean, var = oracle.gp_posterior(X, ls[1], s2[1], L, a, Xc)
    K = _kernel_matrix(X, ls[1], s2[1], noise[1])
    Ks = np.array([[oracle.matern52(c.astype(np.float64), x, ls[1], s2[1]) for x in X] for c in Xc])
    np.testing.assert_allclose(mean, Ks @ np.linalg.solve(K, y), rtol=1e-9, atol=1e-11)
    sol = np.linalg.solve(K, Ks.T)
    np.testing.assert_allclose(var, s2[1] - np.einsum("ij,ji->i", Ks, sol), rtol=1e-8, atol=1e-11)


def test_posterior_interpolates_as_noise_vanishes():
    rng = np.random.default_rng(5)
    X = rng.random((20, 3)).astype(np.float32).astype(np.float64)  # exactly representable
    y = rng.normal(size=20)
    ls = np.full(3, 0.15)
    L, a = _fit(X, y, ls, 1.0, 1e-10)
    mean, var = oracle.gp_posterior(X, ls, 1.0, L, a, X.astype(np.float32))
    np.testing.assert_allclose(mean, y, atol=1e-6)
    assert np.all(var >= 0) and np.all(var < 1e-7)


def test_posterior_bounds_and_far_field():
    w = wl.WORKLOADS[1]
    X, Y = wl.training_set(w, 0)
    ls, s2, noise = wl.hyperparameters(w, 0)
    y = oracle.standardize(Y)[:, 0]
    L, a = _fit(X, y, ls[0], s2[0], noise[0])
    Xc = wl.candidates(w, 0, 0, 500)
    mean, var = oracle.gp_posterior(X, ls[0], s2[0], L, a, Xc)
    assert np.all(var >= 0) and np.all(var <= s2[0])
    far = (Xc[:5] + 1000.0).astype(np.float32)
    mf, vf = oracle.gp_posterior(X, ls[0], s2[0], L, a, far)
    np.testing.assert_allclose(mf, 0.0, atol=1e-300)
    np.testing.assert_allclose(vf, s2[0], rtol=1e-15)


def test_posterior_single_point_closed_form():
    X = np.array([[0.25, 0.5]])
    ls = np.array([0.4, 0.9])
    s2, noise, y = 1.3, 0.2, np.array([0.7])
    L, a = _fit(X, y, ls, s2, noise)
    c = np.array([[0.5, 0.125]], np.float32)
    k = _matern_bessel(np.linalg.norm((c[0].astype(np.float64) - X[0]) / ls), 2.5, s2)
    mean, var = oracle.gp_posterior(X, ls, s2, L, a, c)
    assert mean[0] == pytest.approx(k * y[0] / (s2 + noise), rel=1e-12)
    assert var[0] == pytest.approx(s2 - k * k / (s2 + noise), rel=1e-12)


# ------------------------------------------------------------ Pareto front
def _front_bruteforce(Y, ref):
    n = len(Y)
    keep = np.all(Y < ref, 1)
    for i in range(n):
        le = np.all(Y <= Y[i], 1)
        lt = np.any(Y < Y[i], 1)
        eq = np.all(Y == Y[i], 1)
        if np.any(le & lt) or np.any(eq[:i]):
            keep[i] = False
    return keep


def test_pareto_hand_case():
    Y = np.array([[1, 3], [2, 2], [3, 1], [2, 3], [1, 3], [0, 5], [5, 0]], float)
    mask, order = oracle.pareto_front(Y, np.array([4.0, 4.0]))
    # (2,3) is dominated by (2,2); index 4 duplicates index 0; (0,5), (5,0) lie beyond ref
    assert mask.tolist() == [True, True, True, False, False, False, False]
    assert order.tolist() == [0, 1, 2]


@pytest.mark.parametrize("m", [2, 3])
def test_pareto_invariants_and_bruteforce(m):
    rng = np.random.default_rng(m)
    Y = np.round(rng.normal(size=(300, m)), 1)  # rounding creates ties and duplicates
    ref = np.full(m, 1.1)
    mask, order = oracle.pareto_front(Y, ref)
    assert mask.tolist() == _front_bruteforce(Y, ref).tolist()
    F = Y[order]
    assert sorted(order.tolist()) == np.flatnonzero(mask).tolist()
    assert all(tuple(F[i]) < tuple(F[i + 1]) for i in range(len(F) - 1))  # strictly sorted
    for i in np.flatnonzero(~mask):  # dropped: dominated/duplicated by a kept point, or beyond ref
        if np.all(Y[i] < ref):
            assert np.any(np.all(F <= Y[i], 1))


# ------------------------------------------------------------ hypervolume
def _hv_grid(F, ref):
    """Count unit cells [z, z+1) inside the dominated region (integer data)."""
    F = np.asarray(F, int).reshape(-1, len(ref))
    lo = F.min(0) if len(F) else np.asarray(ref)
    axes = [np.arange(lo[t], ref[t]) for t in range(len(ref))]
    if any(len(a) == 0 for a in axes):
        return 0
    Z = np.stack(np.meshgrid(*axes, indexing="ij"), -1).reshape(-1, len(ref))
    return int(np.any(np.all(F[None, :, :] <= Z[:, None, :], -1), 1).sum())


def test_hv_golden_cases():
    gold = json.load(open(GOLD))
    for case in gold["hv"]:
        assert oracle.hv(case["F"], np.array(case["ref"], float)) == pytest.approx(case["hv"], abs=1e-12)
    for case in gold["hvi"]:
        got = oracle.hvi(case["F"], np.array(case["ref"], float), np.array(case["y"], float))
        assert got == pytest.approx(case["hvi"], abs=1e-12)


@pytest.mark.parametrize("m,seed", [(2, 0), (2, 1), (3, 2), (3, 3), (4, 4)])
def test_hv_matches_grid_enumeration(m, seed):
    rng = np.random.default_rng(seed)
    ref = np.full(m, 8 if m < 4 else 5)
    for _ in range(20):
        F = rng.integers(0, ref[0] + 2, size=(rng.integers(0, 9), m))
        assert oracle.hv(F.astype(float), ref.astype(float)) == _hv_grid(F, ref)
        y = rng.integers(0, ref[0], size=m)
        want = _hv_grid(np.vstack([F, y]), ref) - _hv_grid(F, ref)
        assert oracle.hvi(F.astype(float), ref.astype(float), y.astype(float)) == want


# ------------------------------------------------------------ EHVI (closed form)
def _hvi_staircase_integral(F, ref, y):
    """2-D HVI by integrating, over z1 in [y1, r1), the exposed height
    min(r2, h(z1)) - y2 where h(z1) = min{p2 : p in F, p1 <= z1}."""
    F = np.asarray(F, float).reshape(-1, 2)
    cuts = sorted({y[0], ref[0], *[p[0] for p in F if y[0] < p[0] < ref[0]]})
    tot = 0.0
    for a, b in zip(cuts[:-1], cuts[1:]):
        h = min([ref[1]] + [p[1] for p in F if p[0] <= a])
        tot += (b - a) * max(0.0, h - y[1])
    return tot if y[0] < ref[0] else 0.0


def _front2d(seed, P):
    rng = np.random.default_rng(seed)
    x = np.sort(rng.uniform(-1.5, 0.8, P))
    ys = np.sort(rng.uniform(-1.5, 0.8, P))[::-1]
    return np.stack([x, ys], 1)


def test_ehvi_golden_cases():
    gold = json.load(open(GOLD))
    for case in gold["ehvi2d"]:
        got = oracle.ehvi2d(np.array([case["mean"]]), np.array([case["var"]]),
                            np.array(case["F"], float).reshape(-1, 2), np.array(case["ref"]))
        assert got[0] == pytest.approx(case["ehvi"], rel=1e-14)


def test_ehvi_empty_front_by_quadrature():
    ref = np.array([1.1, 1.1])
    mean = np.array([[0.3, 1.5], [-2.0, 0.9]])
    var = np.array([[0.49, 0.25], [1.7, 0.01]])

    def e_pos(r, mu, s):
        f = lambda y: (r - y) * math.exp(-0.5 * ((y - mu) / s) ** 2) / (s * math.sqrt(2 * math.pi))
        return scipy.integrate.quad(f, mu - 40 * s, r, epsabs=1e-14, epsrel=1e-12, limit=200)[0]

    got = oracle.ehvi2d(mean, var, np.zeros((0, 2)), ref)
    for c in range(2):
        want = e_pos(ref[0], mean[c, 0], math.sqrt(var[c, 0])) * e_pos(ref[1], mean[c, 1],
                                                                        math.sqrt(var[c, 1]))
        assert got[c] == pytest.approx(want, rel=1e-9)


def test_hvi_cell_sum_and_staircase_integral_agree():
    F = _front2d(7, 6)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(8)
    for y in rng.uniform(-2, 1.5, (200, 2)):
        assert oracle.hvi(F, ref, y) == pytest.approx(_hvi_staircase_integral(F, ref, y),
                                                      abs=1e-12)


@pytest.mark.parametrize("case", range(4))
def test_ehvi_matches_brute_force_monte_carlo(case):
    """1e6 samples per candidate; candidates whose EHVI is not a tail event."""
    F = _front2d(11 + case, 6)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(100 + case)
    mu = F.min(0) + rng.uniform(-0.6, 0.3, 2)  # improving on most samples
    sd = rng.uniform(0.08, 0.2, 2)
    got = oracle.ehvi2d(mu[None], (sd ** 2)[None], F, ref)[0]
    n = 1_000_000  # antithetic pairs: z and -z
    Z = rng.standard_normal((n // 2, 2))
    Ysmp = mu + sd * np.concatenate([Z, -Z])
    # vectorised staircase integral of the HVI of every sample
    cuts = np.concatenate([F[:, 0], [ref[0]]])
    lefts = np.concatenate([[-np.inf], F[:, 0]])
    heights = np.concatenate([[ref[1]], F[:, 1]])
    w = np.clip(cuts[None, :] - np.maximum(lefts[None, :], Ysmp[:, :1]), 0, None)
    h = np.clip(heights[None, :] - Ysmp[:, 1:], 0, None)
    mc = (w * h).sum(1)
    se = (0.5 * (mc[:n // 2] + mc[n // 2:])).std() / math.sqrt(n // 2)
    assert se < 3e-4 * got  # the 1e-3 bar is at least 3 standard errors wide
    assert abs(got - mc.mean()) < 1e-3 * got


def test_ehvi_by_2d_quadrature_against_exact_hvi():
    F = _front2d(21, 4)
    ref = np.array([1.1, 1.1])
    mu, sd = np.array([0.0, -0.2]), np.array([0.4, 0.3])
    got = oracle.ehvi2d(mu[None], (sd ** 2)[None], F, ref)[0]
    pdf = lambda y, m, s: math.exp(-0.5 * ((y - m) / s) ** 2) / (s * math.sqrt(2 * math.pi))
    breaks = sorted(set(F[:, 0].tolist() + [ref[0]]))
    tot = 0.0
    lo = mu[0] - 9 * sd[0]
    for a, b in zip([lo] + breaks[:-1], breaks):
        if b <= lo:
            continue
        tot += scipy.integrate.dblquad(
            lambda y2, y1: oracle.hvi(F, ref, np.array([y1, y2])) * pdf(y1, mu[0], sd[0]) *
            pdf(y2, mu[1], sd[1]), max(a, lo), b, mu[1] - 9 * sd[1], ref[1],
            epsabs=1e-10, epsrel=1e-8)[0]
    assert got == pytest.approx(tot, rel=1e-5)


def test_ehvi_limits_and_sign():
    F = _front2d(31, 5)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(32)
    mu = rng.uniform(-2, 2, (300, 2))
    var = rng.uniform(0, 1, (300, 2))
    e = oracle.ehvi2d(mu, var, F, ref)
    assert np.all(e >= 0)
    # sigma -> 0: EHVI -> HVI(mu)
    e0 = oracle.ehvi2d(mu, np.zeros_like(var), F, ref)
    for c in range(300):
        assert e0[c] == pytest.approx(oracle.hvi(F, ref, mu[c]), abs=1e-13)
    e1 = oracle.ehvi2d(mu[:20], np.full((20, 2), 1e-16), F, ref)
    np.testing.assert_allclose(e1, e0[:20], atol=1e-7)
    # a candidate well inside the dominated region with tiny sigma: ~0
    dom = F.max(0) + 0.5
    assert oracle.ehvi2d(dom[None], np.full((1, 2), 1e-4), F, ref)[0] < 1e-12


# ------------------------------------------------------------ MC HVI
@pytest.mark.parametrize("m", [2, 3])
def test_mc_hvi_is_the_sample_mean_of_exact_hvi(m):
    rng = np.random.default_rng(40 + m)
    ref = np.full(m, 1.1)
    Yobs = rng.normal(size=(60, m))
    mask, order = oracle.pareto_front(Yobs, ref)
    F = Yobs[order]
    N, S = 7, 16
    mean = rng.normal(size=(N, m))
    var = rng.uniform(0, 0.5, (N, m))
    eps = rng.standard_normal((N, m, S)).astype(np.float32)
    got = oracle.mc_hvi(mean, var, eps, F, ref)
    for c in range(N):
        ys = mean[c][:, None] + np.sqrt(var[c])[:, None] * eps[c].astype(np.float64)
        want = np.mean([oracle.hvi(F, ref, ys[:, s]) for s in range(S)])
        assert got[c] == pytest.approx(want, rel=1e-12, abs=1e-15)
    # shared normals (candidate stride 0) equal per-candidate copies of the same block
    shared = oracle.mc_hvi(mean, var, eps[:1], F, ref, eps_stride=0)
    rep = oracle.mc_hvi(mean, var, np.repeat(eps[:1], N, 0), F, ref)
    np.testing.assert_allclose(shared, rep, rtol=0, atol=0)


def test_mc_hvi_zero_variance_and_convergence_to_closed_form():
    F = _front2d(51, 5)
    ref = np.array([1.1, 1.1])
    mu = np.array([[-0.3, 0.1], [0.2, -0.6]])
    eps = np.random.default_rng(52).standard_normal((2, 2, 8)).astype(np.float32)
    z = oracle.mc_hvi(mu, np.zeros((2, 2)), eps, F, ref)
    for c in range(2):
        assert z[c] == pytest.approx(oracle.hvi(F, ref, mu[c]), abs=1e-14)
    var = np.array([[0.2, 0.1], [0.05, 0.3]])
    S = 200_000
    eps = np.random.default_rng(53).standard_normal((1, 2, S)).astype(np.float32)
    mc = oracle.mc_hvi(mu, var, eps, F, ref, eps_stride=0)
    cf = oracle.ehvi2d(mu, var, F, ref)
    np.testing.assert_allclose(mc, cf, rtol=1e-2)


# ------------------------------------------------------------ top-k
def test_topk_order_ties_and_nan():
    rng = np.random.default_rng(60)
    acq = np.round(rng.random(5000), 3)  # many ties
    acq[[5, 17, 400]] = np.nan
    acq[[9, 10]] = np.inf
    idx, val = oracle.topk(acq, 64)
    key = np.where(np.isnan(acq), -np.inf, acq)
    ref_order = np.lexsort((np.arange(acq.size), -key))
    assert idx.tolist() == ref_order[:64].tolist()
    assert np.array_equal(val, acq[ref_order[:64]])
    idx_all, _ = oracle.topk(acq, 10**6)  # k > N returns N entries, NaN last
    assert idx_all.tolist() == ref_order.tolist()


# ------------------------------------------------------------ composed step
def test_pipeline_config0_end_to_end_shapes_and_topk_consistency():
    w = wl.WORKLOADS[0]
    X, Y = wl.training_set(w, 0)
    ls, s2, noise = wl.hyperparameters(w, 0)
    fp = pipeline.fit_problem(X, Y, ls, s2, noise, wl.ref_point(w))
    Xc = wl.candidates(w, 0)
    mean, var, acq, idx, val = pipeline.score(fp, Xc, w.mode, w.k)
    assert mean.shape == (w.N, 2) and acq.shape == (w.N,) and idx.shape == (w.k,)
    assert np.all(acq >= 0) and np.all(np.diff(val) <= 0)
    assert fp.front.shape[0] == int(fp.mask.sum())


# ------------------------------------------------------------ constrained acquisition
# Sec. 5.2 "Constrained qNEHVI": the expectation of HVI times the feasibility
# indicator 1[g_t <= 0], g_t = Y_t - c_t on the minimised objectives.
def test_constraints_at_infinity_change_nothing():
    F = _front2d(61, 6)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(62)
    mu = rng.uniform(-2, 2, (50, 2))
    var = rng.uniform(0, 1, (50, 2))
    inf = np.array([np.inf, np.inf])
    np.testing.assert_array_equal(oracle.ehvi2d(mu, var, F, ref, cons=inf),
                                  oracle.ehvi2d(mu, var, F, ref))
    eps = rng.standard_normal((50, 2, 32)).astype(np.float32)
    np.testing.assert_array_equal(oracle.mc_hvi(mu, var, eps, F, ref, cons=inf),
                                  oracle.mc_hvi(mu, var, eps, F, ref))


def test_constrained_ehvi_empty_front_by_quadrature():
    ref = np.array([1.1, 1.1])
    mean = np.array([[0.3, 1.5], [-2.0, 0.9], [0.0, 0.0]])
    var = np.array([[0.49, 0.25], [1.7, 0.01], [0.3, 0.2]])
    cons = np.array([0.4, 2.0])  # the first cuts below r1, the second is above r2

    def e_pos(r, c, mu, s):  # E[(r - Y)_+ 1[Y <= c]] by quadrature over y <= min(r, c)
        f = lambda y: (r - y) * math.exp(-0.5 * ((y - mu) / s) ** 2) / (s * math.sqrt(2 * math.pi))
        return scipy.integrate.quad(f, mu - 40 * s, min(r, c), epsabs=1e-14, epsrel=1e-12,
                                    limit=200)[0]

    got = oracle.ehvi2d(mean, var, np.zeros((0, 2)), ref, cons=cons)
    for c in range(3):
        want = (e_pos(ref[0], cons[0], mean[c, 0], math.sqrt(var[c, 0])) *
                e_pos(ref[1], cons[1], mean[c, 1], math.sqrt(var[c, 1])))
        assert got[c] == pytest.approx(want, rel=1e-9, abs=1e-300)


@pytest.mark.parametrize("case", range(3))
def test_constrained_ehvi_matches_brute_force_monte_carlo(case):
    """1e6 samples per candidate with the feasibility indicator applied."""
    F = _front2d(71 + case, 6)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(170 + case)
    mu = F.min(0) + rng.uniform(-0.6, 0.3, 2)
    sd = rng.uniform(0.08, 0.2, 2)
    cons = mu + sd * rng.uniform(-0.3, 0.8, 2)  # cuts inside each objective's spread
    got = oracle.ehvi2d(mu[None], (sd ** 2)[None], F, ref, cons=cons)[0]
    cuts = np.concatenate([F[:, 0], [ref[0]]])
    lefts = np.concatenate([[-np.inf], F[:, 0]])
    heights = np.concatenate([[ref[1]], F[:, 1]])
    sums = []
    for _ in range(8):  # 8 x 5e5 antithetic pairs
        Z = rng.standard_normal((500_000, 2))
        pair = []
        for Ysmp in (mu + sd * Z, mu - sd * Z):
            w = np.clip(cuts[None, :] - np.maximum(lefts[None, :], Ysmp[:, :1]), 0, None)
            h = np.clip(heights[None, :] - Ysmp[:, 1:], 0, None)
            pair.append((w * h).sum(1) * np.all(Ysmp <= cons, axis=1))
        sums.append(0.5 * (pair[0] + pair[1]))
    mc = np.concatenate(sums)
    se = mc.std() / math.sqrt(mc.size)
    assert se < 1e-3 * got  # resolves errors of a few tenths of a percent
    assert abs(got - mc.mean()) < 4 * se


def test_constrained_ehvi_by_2d_quadrature_against_exact_hvi():
    F = _front2d(81, 4)
    ref = np.array([1.1, 1.1])
    mu, sd = np.array([0.0, -0.2]), np.array([0.4, 0.3])
    cons = np.array([0.1, -0.1])
    got = oracle.ehvi2d(mu[None], (sd ** 2)[None], F, ref, cons=cons)[0]
    pdf = lambda y, m, s: math.exp(-0.5 * ((y - m) / s) ** 2) / (s * math.sqrt(2 * math.pi))
    breaks = sorted(set(F[:, 0].tolist() + [ref[0], cons[0]]))
    tot = 0.0
    lo = mu[0] - 9 * sd[0]
    for a, b in zip([lo] + breaks[:-1], breaks):
        if b <= lo or a >= cons[0]:
            continue
        tot += scipy.integrate.dblquad(
            lambda y2, y1: oracle.hvi(F, ref, np.array([y1, y2])) * pdf(y1, mu[0], sd[0]) *
            pdf(y2, mu[1], sd[1]), max(a, lo), min(b, cons[0]), mu[1] - 9 * sd[1],
            min(ref[1], cons[1]), epsabs=1e-10, epsrel=1e-8)[0]
    assert got == pytest.approx(tot, rel=1e-5)


@pytest.mark.parametrize("m", [2, 3])
def test_constrained_mc_hvi_is_the_sample_mean_of_feasible_hvi(m):
    rng = np.random.default_rng(90 + m)
    ref = np.full(m, 1.1)
    Yobs = rng.normal(size=(60, m))
    mask, order = oracle.pareto_front(Yobs, ref)
    F = Yobs[order]
    N, S = 7, 16
    mean = rng.normal(size=(N, m))
    var = rng.uniform(0, 0.5, (N, m))
    eps = rng.standard_normal((N, m, S)).astype(np.float32)
    cons = rng.uniform(-0.5, 0.8, m)
    got = oracle.mc_hvi(mean, var, eps, F, ref, cons=cons)
    for c in range(N):
        ys = mean[c][:, None] + np.sqrt(var[c])[:, None] * eps[c].astype(np.float64)
        vals = []
        for s in range(S):
            y = ys[:, s]
            hv = _hvi_staircase_integral(F, ref, y) if m == 2 else oracle.hvi(F, ref, y)
            vals.append(hv if np.all(y <= cons) else 0.0)
        assert got[c] == pytest.approx(np.mean(vals), rel=1e-12, abs=1e-15)


def test_constrained_acquisition_limits():
    F = _front2d(95, 5)
    ref = np.array([1.1, 1.1])
    rng = np.random.default_rng(96)
    mu = rng.uniform(-1.5, 1.0, (200, 2))
    var = rng.uniform(0.01, 0.5, (200, 2))
    free = oracle.ehvi2d(mu, var, F, ref)
    prev = np.zeros(200)
    for c in (-40.0, -1.0, -0.3, 0.2, 0.8, 5.0):  # non-decreasing in the thresholds
        e = oracle.ehvi2d(mu, var, F, ref, cons=np.array([c, c]))
        assert np.all(e >= -1e-15) and np.all(e <= free + 1e-12)
        assert np.all(e >= prev - 1e-12)
        prev = e
    assert np.all(oracle.ehvi2d(mu, var, F, ref, cons=np.array([-40.0, 0.0])) < 1e-300)
    np.testing.assert_allclose(prev, free, rtol=1e-12, atol=1e-15)  # c far above every sample


# ------------------------------- composite kernel and outcome transforms (Sec. 5.2, Sec. 6)
def _kc(s2_c, s2_x, beta, pref):
    return np.concatenate([[s2_c, s2_x, beta], np.asarray(pref, np.float64)])


@pytest.mark.parametrize("r", [0.0, 1e-3, 0.3, 1.0, 2.5, 6.0])
def test_matern32_equals_general_matern_at_nu_1p5(r):
    ls = np.array([0.8, 2.0, 1.3])
    u = np.array([-0.4, 0.3, 0.7])
    u = u / np.linalg.norm(u / ls) * r if r > 0 else np.zeros(3)
    a = np.array([1.0, 2.0, 0.5])
    got = oracle.matern32(a, a + u, ls, 0.6)
    assert got == pytest.approx(_matern_bessel(r, 1.5, 0.6), rel=1e-12, abs=1e-300)


def test_preference_weight_hand_values():
    # w(c) = exp(beta <s, a>): allocations (2, 4) with suitabilities (0.5, 0.25)
    assert oracle.pref_weight([2.0, 4.0], 0.1, [0.5, 0.25]) == pytest.approx(math.exp(0.2),
                                                                             rel=1e-15)
    assert oracle.pref_weight([2.0, 4.0], 0.0, [0.5, 0.25]) == 1.0


def test_composite_routing_term_alone_is_matern52_of_the_routing_features():
    rng = np.random.default_rng(21)
    a, b, ls = rng.random(5), rng.random(5), rng.random(5) + 0.3
    kc = _kc(0.0, 0.0, 0.3, [0.2, 0.9])
    got = oracle.kernel(a, b, ls, 1.3, (3, kc))
    assert got == pytest.approx(oracle.matern52(a[:3], b[:3], ls[:3], 1.3), rel=1e-15)
    b2 = b.copy(); b2[3:] += 5.0  # the deployment features do not enter this term
    assert oracle.kernel(a, b2, ls, 1.3, (3, kc)) == pytest.approx(got, rel=1e-15)
    # every feature a routing feature: the plain Matern-5/2 kernel
    assert oracle.kernel(a, b, ls, 1.3, (5, _kc(0.0, 0.0, 0.0, []))) == pytest.approx(
        oracle.kernel(a, b, ls, 1.3), rel=1e-15)


def test_composite_deployment_term_worked_example():
    # k~_c = s2_c w(c) w(c*) k32(c, c*), routing features irrelevant:
    # c = (2, 1), c* = (0, 3), lengthscales (2, 1): r^2 = 1 + 4 = 5;
    # w(c) = exp(0.1 (0.5*2 + 0.25*1)) = exp(0.125), w(c*) = exp(0.075)
    a = np.array([0.3, 2.0, 1.0])
    b = np.array([0.9, 0.0, 3.0])
    ls = np.array([0.5, 2.0, 1.0])
    kc = _kc(0.7, 0.0, 0.1, [0.5, 0.25])
    sr = math.sqrt(3.0 * 5.0)
    want = 0.7 * math.exp(0.2) * (1.0 + sr) * math.exp(-sr)
    assert oracle.kernel(a, b, ls, 0.0, (1, kc)) == pytest.approx(want, rel=1e-14)
    b2 = b.copy(); b2[0] = -4.0
    assert oracle.kernel(a, b2, ls, 0.0, (1, kc)) == pytest.approx(want, rel=1e-14)
    # at zero distance: s2_c w(c)^2
    assert oracle.kernel(a, a, ls, 0.0, (1, kc)) == pytest.approx(0.7 * math.exp(0.25),
                                                                  rel=1e-15)


def test_composite_interaction_term_is_a_product():
    # s2_x alone: k(a, b) = k52(tau, tau*) k32(c, c*), so it factorises into
    # the value with only the routing features moved times the value with
    # only the deployment features moved; each factor is pinned above
    rng = np.random.default_rng(22)
    a, b, ls = rng.random(6), rng.random(6) * 3, rng.random(6) + 0.4
    kc = _kc(0.0, 0.35, 0.2, rng.random(2))
    dt = 4
    ab_tau = np.concatenate([b[:dt], a[dt:]])
    ab_c = np.concatenate([a[:dt], b[dt:]])
    k = lambda u, v: oracle.kernel(u, v, ls, 0.0, (dt, kc))
    assert k(a, b) == pytest.approx(k(a, ab_tau) * k(a, ab_c) / 0.35, rel=1e-13)
    assert k(a, ab_c) == pytest.approx(0.35 * oracle.matern32(a[dt:], b[dt:], ls[dt:]),
                                       rel=1e-14)
    assert k(a, ab_tau) == pytest.approx(0.35 * oracle.matern52(a[:dt], b[:dt], ls[:dt]),
                                         rel=1e-14)


def test_composite_terms_add_with_their_own_scales():
    rng = np.random.default_rng(23)
    a, b, ls = rng.random(5), rng.random(5) * 2, rng.random(5) + 0.3
    pref = rng.random(2)
    k = lambda s2, sc, sx: oracle.kernel(a, b, ls, s2, (3, _kc(sc, sx, 0.15, pref)))
    assert k(1.1, 0.4, 0.07) == pytest.approx(k(1.1, 0, 0) + k(0, 0.4, 0) + k(0, 0, 0.07),
                                              rel=1e-14)


def test_composite_gram_matrix_is_positive_semidefinite():
    rng = np.random.default_rng(24)
    X = np.concatenate([rng.random((60, 3)), rng.integers(0, 5, (60, 4))], 1).astype(float)
    ls = np.array([0.4, 0.5, 0.6, 1.5, 2.0, 1.0, 1.8])
    kc = _kc(0.5, 0.1, 0.05, rng.random(4))
    K = np.array([[oracle.kernel(x, y, ls, 1.0, (3, kc)) for y in X] for x in X])
    np.testing.assert_allclose(K, K.T, rtol=0, atol=0)
    ev = np.linalg.eigvalsh(K)
    assert ev.min() > -1e-12 * ev.max()


def test_composite_posterior_matches_schur_complement_by_library_solve():
    # the pipeline's fit and posterior with the composite kernel and outcome
    # transforms, against a library solve on the same kernel's Gram matrices
    # (prior variance k(x, x), which varies with the preference weight)
    rng = np.random.default_rng(25)
    n, dt, dc = 40, 3, 3
    X = np.concatenate([rng.random((n, dt)), rng.integers(0, 5, (n, dc))], 1).astype(float)
    lat = np.exp(rng.normal(0, 0.5, n))
    qual = 1.0 / (1.0 + np.exp(-rng.normal(0, 1.0, n)))
    Y = np.stack([lat, qual], 1)
    ls = np.tile(np.array([0.4, 0.5, 0.6, 1.5, 2.0, 1.0]), (2, 1))
    s2, noise = np.array([1.0, 0.8]), np.array([1e-3, 2e-3])
    kc = np.stack([_kc(0.5, 0.1, 0.05, rng.random(dc)), _kc(0.3, 0.2, -0.04, rng.random(dc))])
    fp = pipeline.fit_problem(X, Y, ls, s2, noise, np.array([2.0, 2.0]), kernel=(dt, kc),
                              transforms=[1, 6])
    y = oracle.standardize(np.stack([np.log(lat), -np.log(qual / (1 - qual))], 1))
    np.testing.assert_allclose(fp.Ys, y, rtol=1e-12, atol=1e-12)
    Xc = np.concatenate([rng.random((25, dt)), rng.integers(0, 5, (25, dc))], 1)
    Xc = Xc.astype(np.float32)
    mean, var = pipeline.posterior(fp, Xc)
    for t in range(2):
        k = lambda u, v: oracle.kernel(u, v, ls[t], s2[t], (dt, kc[t]))
        K = np.array([[k(u, v) for v in X] for u in X]) + noise[t] * np.eye(n)
        Ks = np.array([[k(c.astype(np.float64), x) for x in X] for c in Xc])
        prior = np.array([k(c.astype(np.float64), c.astype(np.float64)) for c in Xc])
        np.testing.assert_allclose(mean[:, t], Ks @ scipy.linalg.solve(K, y[:, t]), rtol=1e-9,
                                   atol=1e-10)
        sol = scipy.linalg.solve(K, Ks.T)
        np.testing.assert_allclose(var[:, t], prior - np.einsum("ij,ji->i", Ks, sol), rtol=1e-8,
                                   atol=1e-10)
        assert np.all(var[:, t] <= prior + 1e-12)


def test_outcome_transforms():
    rng = np.random.default_rng(26)
    lat = rng.uniform(0.1, 20.0, 30)
    q = rng.uniform(0.01, 0.99, 30)
    Y = np.stack([lat, q, q, 1 - q, lat], 1)
    T = oracle.outcome_transform(Y, [1, 2, 6, 2, 0])
    np.testing.assert_allclose(T[:, 0], np.log(lat), rtol=1e-15)
    np.testing.assert_allclose(T[:, 1], scipy.special.logit(q), rtol=1e-13, atol=1e-15)
    # logit(1 - q) = -logit(q): the negated transform of q equals the plain
    # transform of 1 - q
    np.testing.assert_allclose(T[:, 2], T[:, 3], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(T[:, 2], -T[:, 1], rtol=0, atol=0)
    np.testing.assert_array_equal(T[:, 4], lat)
    # outside the domain: NaN
    bad = oracle.outcome_transform(np.array([[-1.0, 1.5]]), [1, 2])
    assert np.isnan(bad).all()


# --------------------------- hyperparameters by marginal likelihood (Sec. 6)
def _mll_library(X, y, th):
    """log N(y; 0, K) by scipy on the Gram matrix of the (separately pinned)
    Matern-5/2 kernel; th = (log l_1..log l_d, log s2, log noise)."""
    import scipy.stats
    d = X.shape[1]
    ls, s2, noise = np.exp(th[:d]), math.exp(th[d]), math.exp(th[d + 1])
    K = np.array([[oracle.matern52(a, b, ls, s2) for b in X] for a in X]) + noise * np.eye(len(X))
    return scipy.stats.multivariate_normal(np.zeros(len(X)), K).logpdf(y)


def _mll_problem(seed, n=24, d=3):
    rng = np.random.default_rng(seed)
    X = rng.random((n, d))
    y = oracle.standardize((np.sin(3 * X[:, :1]) + X[:, 1:2] ** 2 + 0.05 * rng.normal(size=(n, 1))))
    return X, y[:, 0]


@pytest.mark.parametrize("seed", [0, 1])
def test_mll_equals_library_logpdf(seed):
    X, y = _mll_problem(seed)
    th = np.array([-0.7, 0.2, -0.1, 0.3, math.log(2e-3)])
    got = oracle.gp_mll(X, y, np.exp(th[:3]), math.exp(th[3]), math.exp(th[4]))
    assert got == pytest.approx(_mll_library(X, y, th), rel=1e-11, abs=1e-10)


@pytest.mark.parametrize("seed", [0, 1])
def test_mll_gradient_matches_finite_differences_of_library_logpdf(seed):
    X, y = _mll_problem(seed)
    th = np.array([-0.7, 0.2, -0.1, 0.3, math.log(2e-3)])
    _, g = oracle.gp_mll(X, y, np.exp(th[:3]), math.exp(th[3]), math.exp(th[4]), grad=True)
    h = 1e-5
    for q in range(len(th)):
        e = np.zeros_like(th); e[q] = h
        fd = (_mll_library(X, y, th + e) - _mll_library(X, y, th - e)) / (2 * h)
        assert g[q] == pytest.approx(fd, rel=1e-6, abs=1e-6), q


def test_learner_first_step_and_bounds():
    X, y = _mll_problem(2)
    th0 = np.array([[-0.7, 0.2, -0.1, 0.3, math.log(2e-3)],
                    [20.0, -20.0, 0.0, 50.0, -50.0]])  # the second starts out of bounds
    _, g = oracle.gp_mll(X, y, np.exp(th0[0, :3]), math.exp(th0[0, 3]), math.exp(th0[0, 4]),
                         grad=True)
    lr = 0.05
    th1, _ = oracle.gp_learn(X, y, th0, 1, lr)
    # Adam's first bias-corrected step: lr * g / (|g| + eps)
    np.testing.assert_allclose(th1[0], th0[0] + lr * g / (np.abs(g) + 1e-8), rtol=0, atol=1e-12)
    th_c, _ = oracle.gp_learn(X, y, th0[1:], 0, lr)
    np.testing.assert_allclose(th_c[0], [oracle.LOG_LS_BOUNDS[1], oracle.LOG_LS_BOUNDS[0], 0.0,
                                         oracle.LOG_S2_BOUNDS[1], oracle.LOG_NOISE_BOUNDS[0]])


def test_learner_reaches_the_grid_search_optimum():
    # one feature: a grid over (log l, log s2, log noise) of the library
    # log-likelihood; the learner must end at least as high, near the argmax
    rng = np.random.default_rng(5)
    X = rng.random((20, 1))
    y = oracle.standardize(np.sin(4 * X) + 0.1 * rng.normal(size=(20, 1)))[:, 0]
    grid = [(a, b, c) for a in np.linspace(-2.5, 0.5, 25) for b in np.linspace(-1.5, 2.0, 15)
            for c in np.linspace(-8.0, -1.0, 15)]
    vals = np.array([oracle.gp_mll(X, y, [math.exp(a)], math.exp(b), math.exp(c))
                     for a, b, c in grid])
    best = int(np.argmax(vals))
    assert _mll_library(X, y, np.array(grid[best])) == pytest.approx(vals[best], rel=1e-10)
    th, mll = oracle.gp_learn(X, y, np.array([[-0.5, 0.0, -4.0], [-2.0, 1.0, -2.0]]), 1500, 0.02)
    assert mll.max() >= vals[best] - 1e-3
    r = int(np.argmax(mll))
    assert abs(th[r, 0] - grid[best][0]) < 0.25


def _mll_library_k(X, y, th, dtau, pref):
    """log N(y; 0, K) by scipy on the composite kernel's Gram matrix;
    th = (log l_1..log l_d, log s2, log noise, log s2_c, log s2_x, beta)."""
    import scipy.stats
    d = X.shape[1]
    kc = np.concatenate([[math.exp(th[d + 2]), math.exp(th[d + 3]), th[d + 4]], pref])
    ls, s2, noise = np.exp(th[:d]), math.exp(th[d]), math.exp(th[d + 1])
    K = np.array([[oracle.kernel(a, b, ls, s2, (dtau, kc)) for b in X] for a in X])
    K += noise * np.eye(len(X))
    return scipy.stats.multivariate_normal(np.zeros(len(X)), K).logpdf(y)


def _composite_mll_problem(seed, n=22):
    rng = np.random.default_rng(seed)
    X = np.concatenate([rng.random((n, 2)), rng.integers(0, 5, (n, 2))], 1).astype(float)
    y = oracle.standardize((np.sin(3 * X[:, :1]) + 0.2 * X[:, 2:3] - 0.1 * X[:, 3:4]
                            + 0.05 * rng.normal(size=(n, 1))))[:, 0]
    return X, y, 2, rng.random(2)


def test_composite_mll_and_gradient_match_library():
    X, y, dtau, pref = _composite_mll_problem(30)
    th = np.array([-0.8, -0.3, 0.5, 0.9, 0.1, math.log(2e-3), math.log(0.4), math.log(0.05), 0.2])
    d = X.shape[1]
    kc = np.concatenate([[math.exp(th[d + 2]), math.exp(th[d + 3]), th[d + 4]], pref])
    v, g = oracle.gp_mll(X, y, np.exp(th[:d]), math.exp(th[d]), math.exp(th[d + 1]), grad=True,
                         kernel=(dtau, kc))
    assert v == pytest.approx(_mll_library_k(X, y, th, dtau, pref), rel=1e-11, abs=1e-10)
    h = 1e-5
    for q in range(len(th)):
        e = np.zeros_like(th); e[q] = h
        fd = (_mll_library_k(X, y, th + e, dtau, pref)
              - _mll_library_k(X, y, th - e, dtau, pref)) / (2 * h)
        assert g[q] == pytest.approx(fd, rel=1e-6, abs=1e-6), q


def test_composite_learner_first_step_and_bounds():
    X, y, dtau, pref = _composite_mll_problem(31)
    d = X.shape[1]
    th0 = np.array([[-0.8, -0.3, 0.5, 0.9, 0.1, math.log(2e-3), math.log(0.4), math.log(0.05), 0.2],
                    [0.0, 0.0, 0.0, 0.0, 0.0, -5.0, -20.0, 20.0, 9.0]])
    kc = np.concatenate([[math.exp(th0[0, d + 2]), math.exp(th0[0, d + 3]), th0[0, d + 4]], pref])
    _, g = oracle.gp_mll(X, y, np.exp(th0[0, :d]), math.exp(th0[0, d]), math.exp(th0[0, d + 1]),
                         grad=True, kernel=(dtau, kc))
    lr = 0.05
    th1, _ = oracle.gp_learn(X, y, th0[:1], 1, lr, kernel=(dtau, pref))
    np.testing.assert_allclose(th1[0], th0[0] + lr * g / (np.abs(g) + 1e-8), rtol=0, atol=1e-12)
    th_c, _ = oracle.gp_learn(X, y, th0[1:], 0, lr, kernel=(dtau, pref))
    np.testing.assert_allclose(th_c[0, d + 2:], [oracle.LOG_SC_BOUNDS[0], oracle.LOG_SC_BOUNDS[1],
                                                 oracle.BETA_BOUNDS[1]])
    th2, mll2 = oracle.gp_learn(X, y, th0[:1], 200, lr, kernel=(dtau, pref))
    assert mll2[0] > _mll_library_k(X, y, th0[0], dtau, pref)


# --------------------------------- Monte-Carlo base normals (counter-based generator)
@pytest.mark.parametrize("key,ctr", [((0, 0), (0, 0, 0, 0)), ((123456789, 987654321), (5, 7, 2, 0)),
                                     ((2**64 - 1, 2**63 + 11), (2**64 - 2, 2**64 - 1, 3, 2**62))])
def test_philox_matches_numpy_bit_generator(key, ctr):
    # numpy's Philox (4 x 64-bit, 10 rounds) is the same generator; it
    # advances the counter by one before each block of four words
    bg = np.random.Philox(key=np.array(key, dtype=np.uint64),
                          counter=np.array(ctr, dtype=np.uint64))
    raw = [int(x) for x in bg.random_raw(8)]
    nxt = list(ctr)
    for i in range(4):  # the counter plus one, with carries
        nxt[i] = (nxt[i] + 1) % 2**64
        if nxt[i] != 0:
            break
    assert oracle.philox4x64(nxt, key) == raw[:4]


def test_base_normals_layout_and_distribution():
    eps = oracle.base_normals(7, 2, 3000, 2, 128)
    # the layout: candidate c, objective t, samples 4j..4j+3 from counter (j, c, b m + t, 0)
    w = oracle.philox4x64((5, 17, 1 * 2 + 1, 0), (7, 0))
    u = [((x >> 11) + 0.5) * 2.0 ** -53 for x in w]
    want = [math.sqrt(-2 * math.log(u[0])) * math.cos(2 * math.pi * u[1]),
            math.sqrt(-2 * math.log(u[0])) * math.sin(2 * math.pi * u[1]),
            math.sqrt(-2 * math.log(u[2])) * math.cos(2 * math.pi * u[3]),
            math.sqrt(-2 * math.log(u[2])) * math.sin(2 * math.pi * u[3])]
    np.testing.assert_allclose(eps[1, 17, 1, 20:24], want, rtol=1e-6, atol=1e-7)
    z = eps.astype(np.float64).ravel()
    se = 1 / math.sqrt(z.size)
    assert abs(z.mean()) < 5 * se and abs(z.var() - 1) < 5 * math.sqrt(2) * se
    assert abs((z ** 4).mean() - 3) < 0.05  # normal kurtosis
    # distinct seeds, problems and objectives give different streams
    assert not np.array_equal(eps[0, :, 0], eps[0, :, 1])
    assert not np.array_equal(eps[0], eps[1])
    assert not np.array_equal(oracle.base_normals(8, 1, 10, 2, 8), eps[:1, :10, :, :8])

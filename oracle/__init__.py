"""CPU oracle for the MOBO candidate-scoring step (test infrastructure only).

A plain fp64 C implementation (``boute_oracle.c``) of what the scoring step
computes, written from the paper (Sec. 4.3 problem, Sec. 5.2 MOBO workflow and
constrained qNEHVI, Sec. 6 kernels and outcome transforms), plus this ctypes
wrapper. Only the test suite, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline leg may import it; the CUDA library never does, and the two share
no code.

Parity pins live in ``tests/test_oracle_pins.py`` and, for the noisy
acquisition (joint in-sample draws), ``tests/test_oracle_noisy.py``. Functions
without an independent pin: none.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "boute_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_fp = ctypes.POINTER(ctypes.c_float)
_ip = ctypes.POINTER(ctypes.c_int)
_lp = ctypes.POINTER(ctypes.c_longlong)
_bp = ctypes.POINTER(ctypes.c_ubyte)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C11, OpenMP over candidates)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "boute_oracle.h"))):
        os.makedirs(os.path.dirname(_LIB), exist_ok=True)
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-std=c11", "-O2", "-fopenmp", "-fPIC", "-shared",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        L.bo_standardize.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp]
        L.bo_matern52.argtypes = [_dp, _dp, ctypes.c_int, _dp, ctypes.c_double]
        L.bo_matern52.restype = ctypes.c_double
        L.bo_gp_fit.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                ctypes.c_double, _dp, _dp]
        L.bo_gp_posterior.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                      _dp, _dp, _fp, ctypes.c_longlong, _dp, _dp, ctypes.c_int]
        L.bo_gp_posterior.restype = None
        L.bo_matern32.argtypes = [_dp, _dp, ctypes.c_int, _dp, ctypes.c_double]
        L.bo_matern32.restype = ctypes.c_double
        L.bo_pref_weight.argtypes = [_dp, ctypes.c_int, ctypes.c_double, _dp]
        L.bo_pref_weight.restype = ctypes.c_double
        L.bo_kernel.argtypes = [_dp, _dp, ctypes.c_int, _dp, ctypes.c_double, ctypes.c_int, _dp]
        L.bo_kernel.restype = ctypes.c_double
        L.bo_outcome_transform.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _ip, _dp]
        L.bo_gp_fit_k.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                  ctypes.c_double, ctypes.c_int, _dp, _dp, _dp]
        L.bo_gp_posterior_k.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                        ctypes.c_int, _dp, _dp, _dp, _fp, ctypes.c_longlong, _dp,
                                        _dp, ctypes.c_int]
        L.bo_gp_posterior_k.restype = None
        L.bo_gp_mll.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                ctypes.c_double, _dp]
        L.bo_gp_mll.restype = ctypes.c_double
        L.bo_gp_learn.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_int,
                                  ctypes.c_int, ctypes.c_double, _dp, _dp, _dp]
        L.bo_philox4x64.argtypes = [ctypes.POINTER(ctypes.c_ulonglong),
                                    ctypes.POINTER(ctypes.c_ulonglong),
                                    ctypes.POINTER(ctypes.c_ulonglong)]
        L.bo_philox4x64.restype = None
        L.bo_base_normals.argtypes = [ctypes.c_ulonglong, ctypes.c_int, ctypes.c_longlong,
                                      ctypes.c_int, ctypes.c_int, _fp]
        L.bo_base_normals.restype = None
        L.bo_gp_mll_k.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                  ctypes.c_double, ctypes.c_int, _dp, _dp]
        L.bo_gp_mll_k.restype = ctypes.c_double
        L.bo_gp_learn_k.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, _dp, _dp,
                                    ctypes.c_int, ctypes.c_int, ctypes.c_double, _dp, _dp, _dp]
        L.bo_pareto_front.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp, _bp, _ip]
        L.bo_hv.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp, _dp]
        L.bo_hv.restype = ctypes.c_double
        L.bo_hvi.argtypes = [_dp, ctypes.c_int, ctypes.c_int, _dp, _dp]
        L.bo_hvi.restype = ctypes.c_double
        L.bo_ehvi2d.argtypes = [_dp, _dp, ctypes.c_longlong, _dp, ctypes.c_int, _dp, _dp, _dp,
                                ctypes.c_int]
        L.bo_ehvi2d.restype = None
        L.bo_mc_hvi.argtypes = [_dp, _dp, ctypes.c_longlong, ctypes.c_int, _fp, ctypes.c_int,
                                ctypes.c_longlong, _dp, ctypes.c_int, _dp, _dp, _dp,
                                ctypes.c_int]
        L.bo_mc_hvi.restype = None
        L.bo_joint_draws.argtypes = [_dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_double,
                                     ctypes.c_double, ctypes.c_int, _dp, ctypes.c_double, _fp,
                                     ctypes.c_int, _fp, ctypes.c_longlong, _dp, _dp, _dp, _dp,
                                     ctypes.c_int]
        L.bo_nehvi_mc.argtypes = [_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, _dp, _dp, _dp,
                                  _fp, ctypes.c_longlong, ctypes.c_longlong, _dp, _dp, _dp,
                                  ctypes.c_int]
        L.bo_nehvi_mc.restype = None
        L.bo_topk.argtypes = [_dp, ctypes.c_longlong, ctypes.c_int, _lp, _dp]
        L.bo_topk.restype = None
        L.bo_default_threads.restype = ctypes.c_int
        _lib = L
    return _lib


def _d(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(_dp)


def _f(a):
    a = np.ascontiguousarray(a, dtype=np.float32)
    return a, a.ctypes.data_as(_fp)


class NotPositiveDefinite(ArithmeticError):
    pass


def default_threads() -> int:
    return int(lib().bo_default_threads())


def standardize(Y):
    Y, pY = _d(Y)
    n, m = Y.shape
    out = np.empty_like(Y)
    rc = lib().bo_standardize(pY, n, m, out.ctypes.data_as(_dp))
    if rc:
        raise ValueError(rc)
    return out


def matern52(a, b, ls, s2=1.0) -> float:
    a, pa = _d(a)
    b, pb = _d(b)
    ls, pl = _d(ls)
    return float(lib().bo_matern52(pa, pb, a.size, pl, s2))


def matern32(a, b, ls, s2=1.0) -> float:
    a, pa = _d(a)
    b, pb = _d(b)
    ls, pl = _d(ls)
    return float(lib().bo_matern32(pa, pb, a.size, pl, s2))


def pref_weight(c, beta, pref) -> float:
    c, pc = _d(c)
    pref, pp = _d(pref)
    return float(lib().bo_pref_weight(pc, c.size, float(beta), pp))


def _kern(kernel):
    """kernel: None (Matern-5/2) or (dtau, kc) with kc = [s2_c, s2_x, beta, pref...]."""
    if kernel is None:
        return 0, None, None
    dtau, kc = kernel
    kc, pk = _d(kc)
    return int(dtau), kc, pk


def kernel(a, b, ls, s2=1.0, kernel=None) -> float:
    """The GP's kernel k(a, b): Matern-5/2 (kernel None) or the composite
    kernel (dtau, kc) of Sec. 5.2."""
    a, pa = _d(a)
    b, pb = _d(b)
    ls, pl = _d(ls)
    dtau, kc, pk = _kern(kernel)
    return float(lib().bo_kernel(pa, pb, a.size, pl, float(s2), dtau, pk))


def outcome_transform(Y, codes):
    """Per-objective transforms before Standardize: codes[t] & 3 = 0 identity,
    1 log, 2 logit; bit 4 negates."""
    Y, pY = _d(Y)
    n, m = Y.shape
    codes = np.ascontiguousarray(codes, np.int32)
    out = np.empty_like(Y)
    rc = lib().bo_outcome_transform(pY, n, m, codes.ctypes.data_as(_ip), out.ctypes.data_as(_dp))
    if rc:
        raise ValueError(rc)
    return out


def gp_fit(X, y, ls, s2, noise, kernel=None):
    """Returns (L, alpha); raises NotPositiveDefinite on a failed pivot.
    kernel: None (Matern-5/2) or (dtau, kc), the composite kernel."""
    X, pX = _d(X)
    y, py = _d(y)
    ls, pl = _d(ls)
    n, d = X.shape
    L = np.empty((n, n))
    alpha = np.empty(n)
    dtau, kc, pk = _kern(kernel)
    if kc is None:
        rc = lib().bo_gp_fit(pX, py, n, d, pl, float(s2), float(noise), L.ctypes.data_as(_dp),
                             alpha.ctypes.data_as(_dp))
    else:
        rc = lib().bo_gp_fit_k(pX, py, n, d, pl, float(s2), float(noise), dtau, pk,
                               L.ctypes.data_as(_dp), alpha.ctypes.data_as(_dp))
    if rc == 2:
        raise NotPositiveDefinite("kernel matrix not positive definite")
    if rc:
        raise ValueError(rc)
    return L, alpha


def gp_posterior(X, ls, s2, L, alpha, Xc, threads: int = 0, kernel=None):
    """Posterior mean and variance (fp64) at fp32 candidates Xc (N x d)."""
    X, pX = _d(X)
    ls, pl = _d(ls)
    L, pL = _d(L)
    alpha, pa = _d(alpha)
    Xc, pc = _f(Xc)
    n, d = X.shape
    N = Xc.shape[0]
    mean = np.empty(N)
    var = np.empty(N)
    dtau, kc, pk = _kern(kernel)
    if kc is None:
        lib().bo_gp_posterior(pX, n, d, pl, float(s2), pL, pa, pc, N, mean.ctypes.data_as(_dp),
                              var.ctypes.data_as(_dp), threads)
    else:
        lib().bo_gp_posterior_k(pX, n, d, pl, float(s2), dtau, pk, pL, pa, pc, N,
                                mean.ctypes.data_as(_dp), var.ctypes.data_as(_dp), threads)
    return mean, var


def gp_mll(X, y, ls, s2, noise, grad: bool = False, kernel=None):
    """Log marginal likelihood of the GP (and its gradient when grad): the
    Matern-5/2 kernel, gradient over (log l, log s2, log noise); or the
    composite kernel kernel = (dtau, kc), gradient over (log l, log s2,
    log noise, log s2_c, log s2_x, beta)."""
    X, pX = _d(X)
    y, py = _d(y)
    ls, pl = _d(ls)
    n, d = X.shape
    if kernel is None:
        g = np.empty(d + 2) if grad else None
        v = lib().bo_gp_mll(pX, py, n, d, pl, float(s2), float(noise),
                            None if g is None else g.ctypes.data_as(_dp))
    else:
        dtau, kc, pk = _kern(kernel)
        g = np.empty(d + 5) if grad else None
        v = lib().bo_gp_mll_k(pX, py, n, d, pl, float(s2), float(noise), dtau, pk,
                              None if g is None else g.ctypes.data_as(_dp))
    return (v, g) if grad else v


#: bounds of the learned log-parameters (log l, log s2, log noise)
LOG_LS_BOUNDS = (math.log(1e-3), math.log(1e3))
LOG_S2_BOUNDS = (math.log(1e-3), math.log(1e3))
LOG_NOISE_BOUNDS = (math.log(1e-4), math.log(10.0))


LOG_SC_BOUNDS = (math.log(1e-4), math.log(1e3))
BETA_BOUNDS = (-3.0, 3.0)


def gp_learn(X, y, theta0, iters: int, lr: float, grad: bool = False, kernel=None):
    """Adam ascent on the log marginal likelihood from R starting points
    theta0 (R x (d + 2) log-parameters; with kernel = (dtau, pref), the
    composite kernel, R x (d + 5)). Returns (theta, mll[, grad])."""
    X, pX = _d(X)
    y, py = _d(y)
    th0, pt = _d(np.atleast_2d(theta0))
    n, d = X.shape
    R = th0.shape[0]
    theta = np.empty_like(th0)
    mll = np.empty(R)
    g = np.empty_like(th0) if grad else None
    gp = None if g is None else g.ctypes.data_as(_dp)
    if kernel is None:
        rc = lib().bo_gp_learn(pX, py, n, d, pt, R, int(iters), float(lr),
                               theta.ctypes.data_as(_dp), mll.ctypes.data_as(_dp), gp)
    else:
        pref, pp = _d(kernel[1])
        rc = lib().bo_gp_learn_k(pX, py, n, d, int(kernel[0]), pp, pt, R, int(iters), float(lr),
                                 theta.ctypes.data_as(_dp), mll.ctypes.data_as(_dp), gp)
    if rc:
        raise ValueError(rc)
    return (theta, mll, g) if grad else (theta, mll)


def philox4x64(ctr, key):
    """Philox4x64-10 of a 4-word counter and a 2-word key (4 uint64)."""
    U = ctypes.c_ulonglong
    c, k, o = (U * 4)(*[int(x) for x in ctr]), (U * 2)(*[int(x) for x in key]), (U * 4)()
    lib().bo_philox4x64(c, k, o)
    return [int(x) for x in o]


def base_normals(seed: int, B: int, N: int, m: int, S: int):
    """B x N x m x S fp32 standard normals from the counter-based generator."""
    out = np.empty((B, N, m, S), np.float32)
    lib().bo_base_normals(int(seed), B, N, m, S, out.ctypes.data_as(_fp))
    return out


def pareto_front(Y, ref):
    """Returns (mask (n,) bool, order (P,) int: kept indices sorted lexicographically)."""
    Y, pY = _d(Y)
    ref, pr = _d(ref)
    n, m = Y.shape
    mask = np.zeros(n, np.uint8)
    order = np.zeros(max(n, 1), np.int32)
    P = lib().bo_pareto_front(pY, n, m, pr, mask.ctypes.data_as(_bp), order.ctypes.data_as(_ip))
    return mask.astype(bool), order[:P].astype(np.int64)


def hv(F, ref) -> float:
    F, pF = _d(np.asarray(F, dtype=np.float64).reshape(-1, len(ref)))
    ref, pr = _d(ref)
    return float(lib().bo_hv(pF, F.shape[0], F.shape[1], pr, None))


def hvi(F, ref, y) -> float:
    F, pF = _d(np.asarray(F, dtype=np.float64).reshape(-1, len(ref)))
    ref, pr = _d(ref)
    y, py = _d(y)
    return float(lib().bo_hvi(pF, F.shape[0], F.shape[1], pr, py))


def _cons(cons):
    """Constraint thresholds (one per objective) or None."""
    if cons is None:
        return None, None
    c, pc = _d(cons)
    return c, pc


def ehvi2d(mean, var, F, ref, threads: int = 0, cons=None):
    """mean, var: N x 2; F: P x 2 sorted by f1 ascending; cons: 2 thresholds
    on the minimised objectives (feasibility indicator) or None."""
    mean, pm = _d(mean)
    var, pv = _d(var)
    F, pF = _d(np.asarray(F, dtype=np.float64).reshape(-1, 2))
    ref, pr = _d(ref)
    c, pc = _cons(cons)
    N = mean.shape[0]
    acq = np.empty(N)
    lib().bo_ehvi2d(pm, pv, N, pF, F.shape[0], pr, pc, acq.ctypes.data_as(_dp), threads)
    return acq


def mc_hvi(mean, var, eps, F, ref, eps_stride: int | None = None, threads: int = 0, cons=None):
    """mean, var: N x m; eps: float32 (N, m, S) (or (1, m, S) with eps_stride=0);
    cons: m thresholds on the minimised objectives (feasibility indicator) or None."""
    mean, pm = _d(mean)
    var, pv = _d(var)
    eps, pe = _f(eps)
    m = mean.shape[1]
    S = eps.shape[-1]
    stride = m * S if eps_stride is None else eps_stride
    F, pF = _d(np.asarray(F, dtype=np.float64).reshape(-1, m))
    ref, pr = _d(ref)
    c, pc = _cons(cons)
    N = mean.shape[0]
    acq = np.empty(N)
    lib().bo_mc_hvi(pm, pv, N, m, pe, S, stride, pF, F.shape[0], pr, pc,
                    acq.ctypes.data_as(_dp), threads)
    return acq


# The in-sample jitter of the noisy acquisition, relative to the outputscale:
# the in-sample posterior covariance K_nn - K_nn K^-1 K_nn is singular up to
# rounding wherever the data pin the function down (the paper's qNEHVI
# samples it through a Cholesky factor and leaves the regularisation open).
JOINT_JITTER = 1e-8


def joint_draws(X, y, ls, s2, noise, z, Xc, jitter: float = JOINT_JITTER, threads: int = 0,
                kernel=None):
    """Joint posterior draws of one objective at the observed points and the
    candidates (Sec. 5.2, constrained qNEHVI). z: (S, n) float32 in-sample
    normals. Returns Yin (S, n), mean (N,), cvar (N,), shift (N, S); the
    candidate's draw s is mean + shift[:, s] + sqrt(max(cvar, 0)) eps_s."""
    X, pX = _d(X)
    y, py = _d(y)
    ls, pl = _d(ls)
    z, pz = _f(z)
    Xc, pc = _f(Xc)
    n, d = X.shape
    S = z.shape[0]
    N = Xc.shape[0]
    Yin = np.empty((S, n))
    mean = np.empty(N)
    cvar = np.empty(N)
    shift = np.empty((N, S))
    dtau, kc, pk = _kern(kernel)
    rc = lib().bo_joint_draws(pX, py, n, d, pl, float(s2), float(noise), dtau, pk, float(jitter),
                              pz, S, pc, N, Yin.ctypes.data_as(_dp), mean.ctypes.data_as(_dp),
                              cvar.ctypes.data_as(_dp), shift.ctypes.data_as(_dp), threads)
    if rc == 2:
        raise NotPositiveDefinite("kernel matrix or in-sample covariance not positive definite")
    if rc:
        raise ValueError(rc)
    return Yin, mean, cvar, shift


def nehvi_mc(Yin, mean, cvar, shift, eps, ref, threads: int = 0, cons=None):
    """Noisy MC hypervolume improvement (q = 1). Yin: (S, n, m) in-sample
    draws; mean, cvar: (N, m); shift: (N, m, S); eps: float32 (N, m, S);
    cons: m thresholds on the minimised objectives or None."""
    Yin, pY = _d(Yin)
    mean, pm = _d(mean)
    cvar, pv = _d(cvar)
    shift, ps = _d(shift)
    eps, pe = _f(eps)
    ref, pr = _d(ref)
    c, pcn = _cons(cons)
    S, n, m = Yin.shape
    N = mean.shape[0]
    acq = np.empty(N)
    lib().bo_nehvi_mc(pY, n, m, S, pm, pv, ps, pe, m * S, N, pr, pcn, acq.ctypes.data_as(_dp),
                      threads)
    return acq


def topk(acq, k: int):
    acq, pa = _d(acq)
    k = min(k, acq.size)
    idx = np.empty(k, np.int64)
    val = np.empty(k)
    lib().bo_topk(pa, acq.size, k, idx.ctypes.data_as(_lp), val.ctypes.data_as(_dp))
    return idx, val

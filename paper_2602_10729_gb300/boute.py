"""Thin ctypes binding of libboute (include/boute.h): argument marshalling only.

Every function carries the C entry point's name and forwards torch tensors'
device pointers and the current CUDA stream; all arithmetic runs in the
library's kernels. There is no fallback: if ``libboute.so`` has not been built,
or the device is not sm_103a, calls raise.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

BOUTE_OK, BOUTE_ERR_INVALID_ARG, BOUTE_ERR_NOT_PD, BOUTE_ERR_CUDA = 0, 1, 2, 3
BOUTE_ERR_OOM, BOUTE_ERR_UNSUPPORTED, BOUTE_ERR_TIMEOUT = 4, 5, 6
BOUTE_ACQ_EHVI2D, BOUTE_ACQ_MC_HVI, BOUTE_ACQ_NEHVI = 0, 1, 2
BOUTE_TF_IDENTITY, BOUTE_TF_LOG, BOUTE_TF_LOGIT, BOUTE_TF_NEGATE = 0, 1, 2, 4

#: exported symbols declared in include/boute.h
SYMBOLS = (
    "boute_status_string", "boute_launch_count", "boute_standardize", "boute_gp_create",
    "boute_gp_fit", "boute_gp_status", "boute_gp_free", "boute_gp_posterior",
    "boute_gp_set_precision", "boute_gp_posterior_fp64",
    "boute_gp_set_insample", "boute_gp_insample", "boute_gp_posterior_joint",
    "boute_insample_fronts", "boute_acq_nehvi2d", "boute_bounds_report", "boute_acq_optimize",
    "boute_engine_optimize",
    "boute_pareto_front", "boute_box_decompose", "boute_acq_ehvi", "boute_acq_mc_hvi",
    "boute_select_topk", "boute_select_topk_noalloc", "boute_engine_create", "boute_engine_step",
    "boute_engine_step_async",
    "boute_engine_step_host", "boute_engine_step_host_async", "boute_engine_sync",
    "boute_engine_scores", "boute_engine_set_timing",
    "boute_engine_stage_times", "boute_engine_launches_per_step", "boute_engine_set_constraints",
    "boute_engine_set_outcome_transforms", "boute_engine_set_kernel", "boute_gp_set_kernel",
    "boute_gp_learn", "boute_gp_learn_k", "boute_mobo_run", "boute_base_normals",
    "boute_engine_set_normals", "boute_engine_set_n", "boute_selftest_wait",
    "boute_engine_free",
)
#: stage names of boute_engine_stage_times, in order
STAGES = ("fit", "front", "posterior", "acquisition", "topk")

_lib = None
_vp = ctypes.c_void_p
_i = ctypes.c_int
_ll = ctypes.c_longlong


class MoboConfig(ctypes.Structure):
    """boute_mobo_config."""
    _fields_ = [("mode", ctypes.c_int), ("S", ctypes.c_int), ("max_evals", ctypes.c_int),
                ("patience", ctypes.c_int), ("learn_iters", ctypes.c_int),
                ("learn_lr", ctypes.c_double), ("seed", ctypes.c_ulonglong),
                ("refine_starts", ctypes.c_int), ("refine_steps", ctypes.c_int),
                ("refine_lr", ctypes.c_double)]


#: boute_objective_fn
ObjectiveFn = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.POINTER(ctypes.c_double), ctypes.c_int,
                               ctypes.POINTER(ctypes.c_double), ctypes.c_int, ctypes.c_void_p)


class BouteError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {status_string(code)} ({code})")
        self.code = code


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None):
    """Load libboute.so; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"libboute.so not built ({path}); run __graft_entry__.build()")
    L = ctypes.CDLL(path)
    sig = {
        "boute_status_string": ([_i], ctypes.c_char_p),
        "boute_launch_count": ([], ctypes.c_ulonglong),
        "boute_standardize": ([_vp, _i, _i, _i, _vp, _vp, _vp], _i),
        "boute_gp_create": ([_i, _i, _i, _i, ctypes.POINTER(_vp)], _i),
        "boute_gp_fit": ([_vp, _vp, _vp, _vp, _vp, _vp, _vp], _i),
        "boute_gp_status": ([_vp, _vp], _i),
        "boute_gp_free": ([_vp], None),
        "boute_gp_posterior": ([_vp, _vp, _ll, _vp, _vp, _vp], _i),
        "boute_gp_set_insample": ([_vp, _i], _i),
        "boute_bounds_report": ([_vp], _i),
        "boute_engine_optimize": ([_vp, _vp, _i, _vp, _i, _vp, _vp, _i, ctypes.c_float, _vp, _vp,
                                   _vp, _vp], _i),
        "boute_acq_optimize": ([_vp, _vp, _vp, _vp, _i, _vp, _i, _vp, _i, _vp, _vp, _i,
                                ctypes.c_float, _vp, _vp, _vp, _vp], _i),
        "boute_gp_insample": ([_vp, _vp, _vp, _vp, _vp, _vp, _vp], _i),
        "boute_gp_posterior_joint": ([_vp, _vp, _ll, _vp, _vp, _vp, _vp], _i),
        "boute_insample_fronts": ([_vp, _i, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
        "boute_acq_nehvi2d": ([_vp, _vp, _vp, _i, _ll, _i, _vp, _ll, _vp, _vp, _i, _vp, _vp,
                               _vp], _i),
        "boute_gp_set_precision": ([_vp, _i], _i),
        "boute_gp_posterior_fp64": ([_vp, _vp, _ll, _vp, _vp, _vp], _i),
        "boute_pareto_front": ([_vp, _i, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
        "boute_box_decompose": ([_vp, _vp, _i, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
        "boute_acq_ehvi": ([_vp, _vp, _i, _ll, _vp, _vp, _i, _vp, _vp, _vp, _vp], _i),
        "boute_acq_mc_hvi": ([_vp, _vp, _i, _ll, _i, _vp, _vp, _vp, _i, _vp, _i, _ll, _vp, _vp,
                              _vp], _i),
        "boute_select_topk": ([_vp, _i, _ll, _i, _vp, _vp, _vp], _i),
        "boute_select_topk_noalloc": ([_vp, _i, _ll, _i, _vp, _vp, _vp], _i),
        "boute_engine_create": ([_i, _i, _i, _i, _ll, _i, _i, _i, ctypes.POINTER(_vp)], _i),
        "boute_engine_step": ([_vp] * 11 + [_vp], _i),
        "boute_engine_step_async": ([_vp] * 11 + [_vp], _i),
        "boute_engine_step_host": ([_vp] * 11 + [_vp], _i),
        "boute_engine_step_host_async": ([_vp] * 11 + [_vp], _i),
        "boute_engine_sync": ([_vp, _vp], _i),
        "boute_engine_scores": ([_vp, _vp, _vp, _vp, _vp], _i),
        "boute_engine_set_timing": ([_vp, _i], _i),
        "boute_engine_stage_times": ([_vp, ctypes.POINTER(ctypes.c_float), _i], _i),
        "boute_engine_launches_per_step": ([_vp], _i),
        "boute_engine_set_constraints": ([_vp, _vp], _i),
        "boute_engine_set_outcome_transforms": ([_vp, _vp], _i),
        "boute_engine_set_kernel": ([_vp, _i, _vp], _i),
        "boute_gp_set_kernel": ([_vp, _i, _vp], _i),
        "boute_gp_learn": ([_vp, _vp, _i, _i, _i, _i, _vp, _i, _i, ctypes.c_double, _vp, _vp, _vp,
                            _vp], _i),
        "boute_gp_learn_k": ([_vp, _vp, _i, _i, _i, _i, _i, _vp, _vp, _i, _i, ctypes.c_double, _vp,
                              _vp, _vp, _vp], _i),
        "boute_base_normals": ([ctypes.c_ulonglong, _i, _ll, _i, _i, _vp, _vp], _i),
        "boute_engine_set_normals": ([_vp, ctypes.c_ulonglong], _i),
        "boute_engine_set_n": ([_vp, _i], _i),
        "boute_selftest_wait": ([_i, ctypes.c_ulonglong, _vp], _i),
        "boute_mobo_run": ([ctypes.POINTER(MoboConfig), _i, _i, _vp, _ll, _vp, _vp, _vp, _vp, _i,
                            _vp, _vp, _vp, _vp, _vp, _vp, _i, ObjectiveFn, _vp, _vp, _vp,
                            ctypes.POINTER(_i), ctypes.POINTER(_i)], _i),
        "boute_engine_free": ([_vp], None),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _lib = L
    return L


def status_string(code: int) -> str:
    try:
        return load().boute_status_string(code).decode()
    except Exception:
        return f"status {code}"


def _check(rc: int, where: str):
    if rc != BOUTE_OK:
        raise BouteError(rc, where)


def _p(t, dtype=None, device=True):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    if device and not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    return t.data_ptr()


def _s(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def boute_launch_count() -> int:
    return int(load().boute_launch_count())


def _codes(codes):
    """A host int array of outcome-transform codes (or None)."""
    if codes is None:
        return None
    return (ctypes.c_int * len(codes))(*[int(c) for c in codes])


def boute_standardize(Y, Ys, stream=None, transforms=None):
    """transforms: None or m outcome-transform codes (BOUTE_TF_*)."""
    B, n, m = Y.shape
    _check(load().boute_standardize(_p(Y, torch.float64), B, n, m, _codes(transforms),
                                    _p(Ys, torch.float64), _s(stream)), "boute_standardize")


class Gp:
    """Owner of a boute_gp handle (device factors of B problems x m objectives)."""

    def __init__(self, B: int, n: int, d: int, m: int):
        self.B, self.n, self.d, self.m = B, n, d, m
        h = _vp()
        _check(load().boute_gp_create(B, n, d, m, ctypes.byref(h)), "boute_gp_create")
        self.handle = h

    def free(self):
        if self.handle:
            load().boute_gp_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def boute_gp_create(B, n, d, m) -> Gp:
    return Gp(B, n, d, m)


def boute_gp_fit(gp: Gp, X, Ys, lengthscale, outputscale, noise, stream=None):
    f64 = torch.float64
    _check(load().boute_gp_fit(gp.handle, _p(X, f64), _p(Ys, f64), _p(lengthscale, f64),
                               _p(outputscale, f64), _p(noise, f64), _s(stream)), "boute_gp_fit")


def boute_gp_status(gp: Gp, stream=None) -> int:
    return int(load().boute_gp_status(gp.handle, _s(stream)))


def boute_gp_free(gp: Gp):
    gp.free()


def boute_gp_learn(X, Ys, theta0, iters: int, lr: float, theta, mll, grad=None, stream=None):
    """X: B x n x d, Ys: B x n x m, theta0 / theta / grad: B x m x R x (d + 2),
    mll: B x m x R (fp64 CUDA tensors)."""
    f64 = torch.float64
    B, n, d = X.shape
    m = Ys.shape[2]
    R = theta0.shape[2]
    _check(load().boute_gp_learn(_p(X, f64), _p(Ys, f64), B, n, d, m, _p(theta0, f64), R,
                                 int(iters), float(lr), _p(theta, f64), _p(mll, f64),
                                 _p(grad, f64), _s(stream)), "boute_gp_learn")


def boute_mobo_run(objective, cand, ref, ls, s2, noise, X0, Y0, *, mode=BOUTE_ACQ_EHVI2D, S=0,
                   eps=None, max_evals=50, patience=20, learn_iters=0, learn_lr=0.05,
                   transforms=None, cons=None, d_tau=0, kc=None, seed=0, refine_starts=0,
                   refine_steps=0, refine_lr=0.01):
    """The optimisation loop. objective(x: (d,) float64 array) -> m outcomes.
    cand: N x d; eps: N x m x S (mode MC); ls: m x d, s2, noise: m (initial
    hyperparameters); X0 / Y0: the first observations. Returns a dict with X,
    Y (the n observations), sel (the chosen candidate per iteration), theta
    (the log-hyperparameters of each iteration), ls, s2, noise, kc (final),
    converged. d_tau, kc: the composite kernel (m x (3 + d - d_tau)); mode MC
    with eps None: the engine's own normals drawn from seed."""
    import numpy as np
    cand = np.ascontiguousarray(cand, np.float32)
    N, d = cand.shape
    X0 = np.asarray(X0, np.float64)
    Y0 = np.asarray(Y0, np.float64)
    n0, m = Y0.shape
    X = np.zeros((max_evals, d))
    Y = np.zeros((max_evals, m))
    X[:n0], Y[:n0] = X0, Y0
    ls = np.ascontiguousarray(ls, np.float64).copy()
    s2 = np.ascontiguousarray(s2, np.float64).copy()
    noise = np.ascontiguousarray(noise, np.float64).copy()
    iters = max(max_evals - n0, 1)
    sel = np.zeros(iters, np.int64)
    kc = None if kc is None else np.ascontiguousarray(kc, np.float64).copy()
    theta = np.zeros((iters, m, d + (2 if kc is None else 5)))
    ref = np.ascontiguousarray(ref, np.float64)
    eps = None if eps is None else np.ascontiguousarray(eps, np.float32)
    tf = None if transforms is None else np.ascontiguousarray(transforms, np.int32)
    cs = None if cons is None else np.ascontiguousarray(cons, np.float64)
    errors = []

    def cb(xp, dd, yp, mm, user):
        try:
            y = np.asarray(objective(np.ctypeslib.as_array(xp, (dd,)).copy()), np.float64)
            for t in range(mm):
                yp[t] = float(y[t])
            return 0
        except Exception as exc:  # reported after the loop returns
            errors.append(exc)
            return 1

    fn = ObjectiveFn(cb)
    cfg = MoboConfig(mode, S, max_evals, patience, learn_iters, learn_lr, int(seed),
                     int(refine_starts), int(refine_steps), float(refine_lr))
    n_out, conv = ctypes.c_int(0), ctypes.c_int(0)
    a = lambda v: None if v is None else v.ctypes.data
    rc = load().boute_mobo_run(ctypes.byref(cfg), d, m, a(cand), N, a(eps), a(ref), a(tf), a(cs),
                               int(d_tau), a(kc), a(ls), a(s2), a(noise), a(X), a(Y), n0, fn, None,
                               a(sel), a(theta), ctypes.byref(n_out), ctypes.byref(conv))
    if errors:
        raise errors[0]
    _check(rc, "boute_mobo_run")
    n = n_out.value
    return dict(X=X[:n], Y=Y[:n], sel=sel[:n - n0], theta=theta[:n - n0], ls=ls, s2=s2,
                noise=noise, kc=kc, converged=bool(conv.value))


def boute_gp_learn_k(X, Ys, d_tau, pref, theta0, iters: int, lr: float, theta, mll, grad=None,
                     stream=None):
    """The composite kernel's learner: pref B x m x (d - d_tau); theta0 /
    theta / grad B x m x R x (d + 5) (fp64 CUDA tensors)."""
    f64 = torch.float64
    B, n, d = X.shape
    m = Ys.shape[2]
    R = theta0.shape[2]
    _check(load().boute_gp_learn_k(_p(X, f64), _p(Ys, f64), B, n, d, m, int(d_tau), _p(pref, f64),
                                   _p(theta0, f64), R, int(iters), float(lr), _p(theta, f64),
                                   _p(mll, f64), _p(grad, f64), _s(stream)), "boute_gp_learn_k")


def boute_base_normals(seed: int, eps, stream=None):
    """Fills eps (B x N x m x S fp32 CUDA tensor) from the counter-based generator."""
    B, N, m, S = eps.shape
    _check(load().boute_base_normals(int(seed), B, N, m, S, _p(eps, torch.float32), _s(stream)),
           "boute_base_normals")


def boute_engine_set_normals(e: Engine, seed: int):
    """The engine's own base normals; steps then take eps=None."""
    _check(load().boute_engine_set_normals(e.handle, int(seed)), "boute_engine_set_normals")


def boute_engine_set_n(e: Engine, n: int):
    """Later steps use n <= the engine's creation n observations."""
    _check(load().boute_engine_set_n(e.handle, int(n)), "boute_engine_set_n")
    e.n = int(n)


def boute_acq_optimize(gp: Gp, lower, upper, K, box_cap, eps, S, X0, P, xlo, xhi, steps, lr, X,
                       acq, grad=None, stream=None):
    """Projected Adam ascent on the 2-objective sample-average MC acquisition
    (CUDA tensors: X0, X B x P x d; acq B x P; grad B x P x d or None)."""
    f32 = torch.float32
    _check(load().boute_acq_optimize(gp.handle, _p(lower, f32), _p(upper, f32),
                                     _p(K, torch.int32), int(box_cap), _p(eps, f32), int(S),
                                     _p(X0, f32), int(P), _p(xlo, f32), _p(xhi, f32), int(steps),
                                     float(lr), _p(X, f32), _p(acq, f32), _p(grad, f32),
                                     _s(stream)), "boute_acq_optimize")


def boute_engine_optimize(e: Engine, eps, S, X0, P, xlo, xhi, steps, lr, X, acq, grad=None,
                          stream=None):
    """boute_acq_optimize on the engine's last step (fit and observed front)."""
    f32 = torch.float32
    _check(load().boute_engine_optimize(e.handle, _p(eps, f32), int(S), _p(X0, f32), int(P),
                                        _p(xlo, f32), _p(xhi, f32), int(steps), float(lr),
                                        _p(X, f32), _p(acq, f32), _p(grad, f32), _s(stream)),
           "boute_engine_optimize")


def boute_bounds_report():
    """Debug build: (unit, line, index, extent) of the first index found outside
    its extent since the last call, or None; raises on the product library."""
    rec = (ctypes.c_longlong * 4)()
    rc = load().boute_bounds_report(rec)
    if rc not in (0, 1):
        raise BouteError(rc, "boute_bounds_report")
    return tuple(rec) if rc == 1 else None


def boute_selftest_wait(complete: bool, limit_ns: int, stream=None) -> int:
    """Status of one bounded device-side wait (BOUTE_ERR_TIMEOUT if it ran out)."""
    return int(load().boute_selftest_wait(int(complete), int(limit_ns), _s(stream)))


def _host_f64(a):
    import numpy as np
    return None if a is None else torch.as_tensor(np.ascontiguousarray(a, np.float64))


def boute_gp_set_kernel(gp: Gp, d_tau: int = 0, params=None):
    """params: None (Matern-5/2) or B x m x (3 + d - d_tau) host values
    [s2_c, s2_x, beta, preference entries...] of the composite kernel."""
    p = _host_f64(params)
    _check(load().boute_gp_set_kernel(gp.handle, int(d_tau), _p(p, torch.float64, False)),
           "boute_gp_set_kernel")


def boute_gp_posterior(gp: Gp, Xc, N: int, mean, var, stream=None):
    f32 = torch.float32
    _check(load().boute_gp_posterior(gp.handle, _p(Xc, f32), N, _p(mean, f32), _p(var, f32),
                                     _s(stream)), "boute_gp_posterior")


BOUTE_PREC_FP32, BOUTE_PREC_FP64 = 0, 1


def boute_gp_set_insample(gp: Gp, S: int):
    """S in-sample joint draws for the noisy acquisition (0: off); fit again after."""
    _check(load().boute_gp_set_insample(gp.handle, int(S)), "boute_gp_set_insample")


def boute_gp_insample(gp: Gp, Ys, outputscale, noise, z, Yin, stream=None):
    """After boute_gp_fit: z (B x m x S x n fp32) in, Yin (same shape) out."""
    f64, f32 = torch.float64, torch.float32
    _check(load().boute_gp_insample(gp.handle, _p(Ys, f64), _p(outputscale, f64),
                                    _p(noise, f64), _p(z, f32), _p(Yin, f32), _s(stream)),
           "boute_gp_insample")


def boute_gp_posterior_joint(gp: Gp, Xc, N: int, mean, cvar, shift, stream=None):
    """mean, cvar: B x m x N; shift: B x m x S x N (fp32 CUDA tensors)."""
    f32 = torch.float32
    _check(load().boute_gp_posterior_joint(gp.handle, _p(Xc, f32), N, _p(mean, f32),
                                           _p(cvar, f32), _p(shift, f32), _s(stream)),
           "boute_gp_posterior_joint")


def boute_insample_fronts(Yin, B, n, S, ref, strips, counts, stream=None, cons=None):
    """Yin: B x 2 x S x n; strips: B x S x (n + 1) x 4 fp32; counts: B x S int32."""
    _check(load().boute_insample_fronts(_p(Yin, torch.float32), B, n, S, _p(ref, torch.float64),
                                        _p(cons, torch.float64), _p(strips, torch.float32),
                                        _p(counts, torch.int32), _s(stream)),
           "boute_insample_fronts")


def boute_acq_nehvi2d(mean, cvar, shift, B, N, S, eps, eps_cand_stride, strips, counts, n, acq,
                      stream=None, cons=None):
    f32 = torch.float32
    _check(load().boute_acq_nehvi2d(_p(mean, f32), _p(cvar, f32), _p(shift, f32), B, N, S,
                                    _p(eps, f32), eps_cand_stride, _p(strips, f32),
                                    _p(counts, torch.int32), n, _p(cons, torch.float64),
                                    _p(acq, f32), _s(stream)), "boute_acq_nehvi2d")


def boute_gp_set_precision(gp: Gp, prec: int):
    _check(load().boute_gp_set_precision(gp.handle, int(prec)), "boute_gp_set_precision")


def boute_gp_posterior_fp64(gp: Gp, Xc, N: int, mean, var, stream=None):
    f64 = torch.float64
    _check(load().boute_gp_posterior_fp64(gp.handle, _p(Xc, torch.float32), N, _p(mean, f64),
                                          _p(var, f64), _s(stream)), "boute_gp_posterior_fp64")


def boute_pareto_front(Ys, B, n, m, ref, mask, front, P, stream=None):
    f64 = torch.float64
    _check(load().boute_pareto_front(_p(Ys, f64), B, n, m, _p(ref, f64), _p(mask, torch.uint8),
                                     _p(front, f64), _p(P, torch.int32), _s(stream)),
           "boute_pareto_front")


def boute_box_decompose(front, P, B, n, m, ref, lower, upper, K, stream=None):
    _check(load().boute_box_decompose(_p(front, torch.float64), _p(P, torch.int32), B, n, m,
                                      _p(ref, torch.float64), _p(lower, torch.float32),
                                      _p(upper, torch.float32), _p(K, torch.int32), _s(stream)),
           "boute_box_decompose")


def boute_acq_ehvi(mean, var, B, N, front, P, n, ref, acq, stream=None, cons=None):
    """cons: None or a B x 2 fp64 CUDA tensor of thresholds (constrained EHVI)."""
    f32, f64 = torch.float32, torch.float64
    _check(load().boute_acq_ehvi(_p(mean, f32), _p(var, f32), B, N, _p(front, f64),
                                 _p(P, torch.int32), n, _p(ref, f64), _p(cons, f64),
                                 _p(acq, f32), _s(stream)), "boute_acq_ehvi")


def boute_acq_mc_hvi(mean, var, B, N, m, lower, upper, K, box_cap, eps, S, eps_cand_stride, acq,
                     stream=None, cons=None):
    """cons: None or a B x m fp64 CUDA tensor of thresholds (constrained MC HVI)."""
    f32 = torch.float32
    _check(load().boute_acq_mc_hvi(_p(mean, f32), _p(var, f32), B, N, m, _p(lower, f32),
                                   _p(upper, f32), _p(K, torch.int32), box_cap, _p(eps, f32), S,
                                   eps_cand_stride, _p(cons, torch.float64), _p(acq, f32),
                                   _s(stream)), "boute_acq_mc_hvi")


def boute_select_topk(acq, B, N, k, idx, val, stream=None):
    _check(load().boute_select_topk(_p(acq, torch.float32), B, N, k, _p(idx, torch.int64),
                                    _p(val, torch.float32), _s(stream)), "boute_select_topk")


def boute_select_topk_noalloc(acq, B, N, k, idx, val, stream=None):
    _check(load().boute_select_topk_noalloc(_p(acq, torch.float32), B, N, k,
                                            _p(idx, torch.int64), _p(val, torch.float32),
                                            _s(stream)), "boute_select_topk_noalloc")


#: bytes of the fixed scratch array behind boute_select_topk_noalloc
TOPK_NOALLOC_SCRATCH_BYTES = 8 << 20


class Engine:
    """Owner of a boute_engine (all buffers of one scoring-step shape)."""

    def __init__(self, B, n, d, m, N, mode, S, k):
        self.B, self.n, self.d, self.m, self.N, self.mode, self.S, self.k = (
            B, n, d, m, N, mode, S, k)
        self.ncap = n
        h = _vp()
        _check(load().boute_engine_create(B, n, d, m, N, mode, S, k, ctypes.byref(h)),
               "boute_engine_create")
        self.handle = h

    def free(self):
        if self.handle:
            load().boute_engine_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def boute_engine_create(B, n, d, m, N, mode, S, k) -> Engine:
    return Engine(B, n, d, m, N, mode, S, k)


def _engine_args(X, Y, ls, s2, noise, ref, Xc, eps, idx, val, device):
    f64, f32 = torch.float64, torch.float32
    return (_p(X, f64, device), _p(Y, f64, device), _p(ls, f64, device), _p(s2, f64, device),
            _p(noise, f64, device), _p(ref, f64, device), _p(Xc, f32, device),
            _p(eps, f32, device), _p(idx, torch.int64, device), _p(val, f32, device))


def boute_engine_step(e: Engine, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, stream=None):
    """Device tensors in and out; synchronises; raises on a fit or device error."""
    _check(load().boute_engine_step(e.handle, *_engine_args(X, Y, ls, s2, noise, ref, Xc, eps,
                                                            idx, val, True), _s(stream)),
           "boute_engine_step")


def boute_engine_step_async(e: Engine, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, stream=None):
    _check(load().boute_engine_step_async(e.handle, *_engine_args(
        X, Y, ls, s2, noise, ref, Xc, eps, idx, val, True), _s(stream)), "boute_engine_step_async")


def boute_engine_step_host(e: Engine, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, stream=None):
    """HOST (CPU, ideally pinned) tensors in and out; copies inside the call."""
    _check(load().boute_engine_step_host(e.handle, *_engine_args(
        X, Y, ls, s2, noise, ref, Xc, eps, idx, val, False), _s(stream)), "boute_engine_step_host")


def boute_engine_step_host_async(e: Engine, X, Y, ls, s2, noise, ref, Xc, eps, idx, val,
                                 stream=None):
    """As boute_engine_step_host without the final synchronisation; the host
    tensors must stay as they are (inputs) and unread (idx, val) until
    boute_engine_sync."""
    _check(load().boute_engine_step_host_async(e.handle, *_engine_args(
        X, Y, ls, s2, noise, ref, Xc, eps, idx, val, False), _s(stream)),
        "boute_engine_step_host_async")


def boute_engine_sync(e: Engine, stream=None):
    _check(load().boute_engine_sync(e.handle, _s(stream)), "boute_engine_sync")


def boute_engine_scores(e: Engine, acq=None, mean=None, var=None, stream=None):
    f32 = torch.float32
    _check(load().boute_engine_scores(e.handle, _p(acq, f32), _p(mean, f32), _p(var, f32),
                                      _s(stream)), "boute_engine_scores")


TIMING_OFF, TIMING_SERIAL, TIMING_LIVE = 0, 1, 2


def boute_engine_set_timing(e: Engine, on=True):
    """on: False/0 off, True/1 serialised stages, 2 live (normal schedule)."""
    _check(load().boute_engine_set_timing(e.handle, int(on)), "boute_engine_set_timing")


def boute_engine_stage_times(e: Engine) -> dict:
    ms = (ctypes.c_float * len(STAGES))()
    _check(load().boute_engine_stage_times(e.handle, ms, len(STAGES)), "boute_engine_stage_times")
    return dict(zip(STAGES, (float(x) for x in ms)))


def boute_engine_launches_per_step(e: Engine) -> int:
    return int(load().boute_engine_launches_per_step(e.handle))


def boute_engine_set_kernel(e: Engine, d_tau: int = 0, params=None):
    """As boute_gp_set_kernel, for the engine's steps."""
    p = _host_f64(params)
    _check(load().boute_engine_set_kernel(e.handle, int(d_tau), _p(p, torch.float64, False)),
           "boute_engine_set_kernel")


def boute_engine_set_outcome_transforms(e: Engine, codes=None):
    """codes: None or m outcome-transform codes (BOUTE_TF_*)."""
    _check(load().boute_engine_set_outcome_transforms(e.handle, _codes(codes)),
           "boute_engine_set_outcome_transforms")


def boute_engine_set_constraints(e: Engine, cons=None):
    """cons: None (unconstrained) or a contiguous B x m fp64 CPU tensor of
    thresholds on the standardised, minimised outcomes (the units of ref)."""
    _check(load().boute_engine_set_constraints(e.handle, _p(cons, torch.float64, False)),
           "boute_engine_set_constraints")


def boute_engine_free(e: Engine):
    e.free()

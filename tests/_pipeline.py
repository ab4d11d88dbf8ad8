"""Test helpers: run the scoring step through the C-ABI one entry point at a
time (so every intermediate can be compared), and the oracle on the same
seeded inputs. The tolerances live here, with their derivation."""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

import oracle
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

# ---- tolerances ----------------------------------------------------------------
# Posterior (fp16 hi/lo contraction with fp32 accumulate, fp32-accurate):
# relative 1e-5 against the quantity's natural scale: |g - o| <= 1e-5 *
# max(|o|, s) for the mean (s is the prior standard deviation), |g - o| <=
# 1e-5 * s2 for the variance, whose fp32 value s2 - ||v||^2 carries an
# absolute rounding error of order eps32 * s2 whatever its size (near a
# training point, where the variance is about the noise, a relative bound on
# the variance itself would ask for digits an fp32 difference cannot keep).
POST_REL = 1e-5
# Acquisition: relative 1e-4 against max(|o|, 1e-3 * max_j |o_j|), the largest
# value of the problem setting the scale below which fp32 rounding of the
# O(1) terms dominates.
ACQ_REL = 1e-4
ACQ_FLOOR = 1e-3


def check_mean(g, o, s2, rel=POST_REL):
    g, o = np.asarray(g, np.float64), np.asarray(o, np.float64)
    s = np.sqrt(np.asarray(s2, np.float64))
    err = np.abs(g - o) / np.maximum(np.abs(o), s)
    assert np.all(np.isfinite(g)), "non-finite posterior mean"
    assert err.max() <= rel, f"mean rel err {err.max():.3g} at {np.argmax(err)}"
    return float(err.max())


def check_var(g, o, s2, rel=POST_REL):
    g, o = np.asarray(g, np.float64), np.asarray(o, np.float64)
    err = np.abs(g - o) / np.asarray(s2, np.float64)
    assert np.all(np.isfinite(g)) and np.all(g >= 0), "bad posterior variance"
    assert err.max() <= rel, f"var rel err {err.max():.3g} at {np.argmax(err)}"
    return float(err.max())


def acq_err(g, o, scale=None):
    g, o = np.asarray(g, np.float64), np.asarray(o, np.float64)
    scale = np.abs(o).max() if scale is None else scale
    return np.abs(g - o) / np.maximum(np.abs(o), ACQ_FLOOR * max(scale, 1e-300))


def check_acq(g, o, rel=ACQ_REL, scale=None):
    e = acq_err(g, o, scale)
    assert np.all(np.isfinite(g)), "non-finite acquisition"
    assert e.max() <= rel, f"acq rel err {e.max():.3g} at {np.argmax(e)} (g={g[np.argmax(e)]}, o={o[np.argmax(e)]})"
    return float(e.max())


def acq_sensitivity(fn, mean, var, s2):
    """First-order change of the oracle acquisition fn(mean, var) (N x m each)
    when every posterior input moves by its tolerance: the part of an
    end-to-end acquisition difference the posterior tolerance accounts for."""
    base = fn(mean, var)
    s2 = np.asarray(s2, np.float64)
    tot = np.zeros_like(base)
    for t in range(mean.shape[1]):
        dm = POST_REL * np.maximum(np.abs(mean[:, t]), np.sqrt(s2[t]))
        dv = POST_REL * s2[t]
        worst_m = np.zeros_like(base)
        worst_v = np.zeros_like(base)
        for sign in (1.0, -1.0):
            mm = mean.copy()
            mm[:, t] += sign * dm
            worst_m = np.maximum(worst_m, np.abs(fn(mm, var) - base))
            vv = var.copy()
            vv[:, t] = np.maximum(vv[:, t] + sign * dv, 0.0)
            worst_v = np.maximum(worst_v, np.abs(fn(mean, vv) - base))
        tot += worst_m + worst_v
    return base, tot


def check_acq_end_to_end(g_acq, fn, mean_g, var_g, mean_o, var_o, s2):
    """(1) the acquisition kernel's own error: GPU acquisition against the
    oracle acquisition of the GPU posterior; (2) against the oracle's own
    acquisition, allowing for the posterior tolerance (acq_sensitivity)."""
    a_at_g = fn(np.asarray(mean_g, np.float64), np.asarray(var_g, np.float64))
    e1 = check_acq(g_acq, a_at_g)
    o, sens = acq_sensitivity(fn, mean_o, var_o, s2)
    scale = np.abs(o).max()
    tol = ACQ_REL * np.maximum(np.abs(o), ACQ_FLOOR * scale) + 2 * sens
    err = np.abs(np.asarray(g_acq, np.float64) - o)
    assert np.all(err <= tol), f"acq e2e err {err.max():.3g} > tol at {np.argmax(err - tol)}"
    return e1, o, tol


def check_topk_consistent(idx_g, acq_o, k, tol_abs):
    """End-to-end top-k: the GPU may differ from the oracle only among
    candidates whose oracle values are within tol_abs of the k-th value."""
    order = np.lexsort((np.arange(acq_o.size), -acq_o))
    kth = acq_o[order[k - 1]]
    sel = set(int(i) for i in idx_g)
    must = {int(i) for i in order[:k] if acq_o[i] > kth + tol_abs}
    assert must <= sel, f"missing clear winners {sorted(must - sel)[:5]}"
    for i in sel:
        assert acq_o[i] >= kth - tol_abs, f"selected {i} with oracle {acq_o[i]} < kth {kth}"


def check_topk_consistent_tol(idx_g, acq_o, k, tol):
    """As check_topk_consistent with a per-candidate tolerance array."""
    order = np.lexsort((np.arange(acq_o.size), -acq_o))
    kth = acq_o[order[k - 1]]
    sel = set(int(i) for i in idx_g)
    must = {int(i) for i in order[:k] if acq_o[i] - tol[i] > kth + tol[order[k - 1]]}
    assert must <= sel, f"missing clear winners {sorted(must - sel)[:5]}"
    for i in sel:
        assert acq_o[i] + tol[i] >= kth - tol[order[k - 1]], f"selected {i} below the k-th"


# ---- workload on the host -------------------------------------------------------
@dataclass
class HostProblem:
    w: wl.Workload
    X: np.ndarray  # B x n x d
    Y: np.ndarray  # B x n x m (raw)
    ls: np.ndarray  # B x m x d
    s2: np.ndarray  # B x m
    noise: np.ndarray  # B x m
    ref: np.ndarray  # B x m
    Xc: np.ndarray  # B x N x d float32
    eps: np.ndarray | None  # B x N x m x S float32
    d_tau: int = 0  # composite kernel: routing features [0, d_tau), kc below
    kc: np.ndarray | None = None  # B x m x (3 + d - d_tau) composite-kernel parameters
    transforms: tuple = ()  # outcome-transform codes per objective

    def kernel(self, b: int):
        """The oracle's kernel argument for problem b."""
        return None if self.kc is None else (self.d_tau, self.kc[b])


def host_problem(w: wl.Workload, N: int | None = None, threads: int = 8) -> HostProblem:
    N = w.N if N is None else N
    Xs, Ys, L, S2, NZ = [], [], [], [], []
    for b in range(w.B):
        X, Y = wl.training_set(w, b)
        ls, s2, nz = wl.hyperparameters(w, b)
        Xs.append(X); Ys.append(Y); L.append(ls); S2.append(s2); NZ.append(nz)
    Xc = np.stack([wl.candidates(w, b, 0, N, threads) for b in range(w.B)])
    eps = None
    if w.mode in ("mc", "nehvi"):
        eps = np.stack([wl.base_normals(w, b, 0, N, threads) for b in range(w.B)])
    ref = np.tile(wl.ref_point(w), (w.B, 1))
    kc = None
    if w.d_tau:
        kc = np.stack([wl.kernel_params(w, b)[1] for b in range(w.B)])
    return HostProblem(w, np.stack(Xs), np.stack(Ys), np.stack(L), np.stack(S2), np.stack(NZ),
                       ref, Xc, eps, w.d_tau, kc, tuple(w.transforms))


def oracle_fit(hp: HostProblem, b: int) -> opl.FittedProblem:
    return opl.fit_problem(hp.X[b], hp.Y[b], hp.ls[b], hp.s2[b], hp.noise[b], hp.ref[b],
                           kernel=hp.kernel(b), transforms=hp.transforms or None)


# ---- GPU: one ABI call at a time ------------------------------------------------
def gpu_pipeline(hp: HostProblem, N: int | None = None, mean_var_in=None, cons=None):
    """Runs standardise -> fit -> front -> boxes -> posterior -> acq -> top-k
    through the C-ABI and returns every intermediate on the host.
    mean_var_in: optional (mean, var) B x m x N float32 fed to the
    acquisition instead of the GPU posterior (isolated acquisition test).
    cons: optional B x m thresholds (constrained acquisition)."""
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = hp.w
    B, n, d, m = w.B, w.n, w.d, w.m
    N = hp.Xc.shape[1] if N is None else N
    dev = torch.device("cuda")
    t = lambda a, dt=None: torch.as_tensor(np.ascontiguousarray(a), device=dev, dtype=dt)
    X, Y = t(hp.X, torch.float64), t(hp.Y, torch.float64)
    ls, s2, nz, ref = (t(hp.ls, torch.float64), t(hp.s2, torch.float64),
                       t(hp.noise, torch.float64), t(hp.ref, torch.float64))
    Xc = t(hp.Xc[:, :N], torch.float32)
    Ys = torch.empty_like(Y)
    bt.boute_standardize(Y, Ys, transforms=hp.transforms or None)
    gp = bt.boute_gp_create(B, n, d, m)
    if hp.kc is not None:
        bt.boute_gp_set_kernel(gp, hp.d_tau, hp.kc)
    bt.boute_gp_fit(gp, X, Ys, ls, s2, nz)
    st = bt.boute_gp_status(gp)
    mask = torch.empty((B, n), dtype=torch.uint8, device=dev)
    front = torch.zeros((B, n, m), dtype=torch.float64, device=dev)
    P = torch.empty(B, dtype=torch.int32, device=dev)
    bt.boute_pareto_front(Ys, B, n, m, ref, mask, front, P)
    mean = torch.empty((B, m, N), dtype=torch.float32, device=dev)
    var = torch.empty_like(mean)
    out = dict(status=st, Ys=Ys.cpu().numpy(), mask=mask.cpu().numpy().astype(bool),
               front=front.cpu().numpy(), P=P.cpu().numpy())
    if st != 0:
        gp.free()
        return out
    bt.boute_gp_posterior(gp, Xc, N, mean, var)
    if mean_var_in is not None:
        mi, vi = (t(a, torch.float32) for a in mean_var_in)
    else:
        mi, vi = mean, var
    acq = torch.empty((B, N), dtype=torch.float32, device=dev)
    cap = 2 * n + 2
    cn = None if cons is None else t(cons, torch.float64)
    if w.mode == "ehvi":
        bt.boute_acq_ehvi(mi, vi, B, N, front, P, n, ref, acq, cons=cn)
    else:
        lower = torch.empty((B, cap, m), dtype=torch.float32, device=dev)
        upper = torch.empty_like(lower)
        K = torch.empty(B, dtype=torch.int32, device=dev)
        bt.boute_box_decompose(front, P, B, n, m, ref, lower, upper, K)
        eps = t(hp.eps[:, :N], torch.float32)
        bt.boute_acq_mc_hvi(mi, vi, B, N, m, lower, upper, K, cap, eps, w.S, m * w.S, acq,
                            cons=cn)
        out.update(lower=lower.cpu().numpy(), upper=upper.cpu().numpy(), K=K.cpu().numpy())
    k = min(w.k, N)
    idx = torch.empty((B, k), dtype=torch.int64, device=dev)
    val = torch.empty((B, k), dtype=torch.float32, device=dev)
    bt.boute_select_topk(acq, B, N, k, idx, val)
    torch.cuda.synchronize()
    out.update(mean=mean.cpu().numpy(), var=var.cpu().numpy(), acq=acq.cpu().numpy(),
               idx=idx.cpu().numpy(), val=val.cpu().numpy(), status=bt.boute_gp_status(gp))
    gp.free()
    return out

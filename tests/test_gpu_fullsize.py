"""The five workloads at full size, through the C-ABI engine in the launch
configuration bench.py times. The oracle recomputes sampled candidates one
by one (contiguous runs including the first and the ragged last tile, plus
the GPU's selections); top-k is checked by properties that hold at any size,
and against the oracle's own selection over every candidate that could
compete for it (the GPU's top-k and every candidate whose GPU score lies
within a few acquisition tolerances of the k-th): the two index sets agree
except for near-ties, candidates whose oracle scores lie within the
tolerance of the oracle's k-th."""
import numpy as np
import pytest

from _pipeline import (ACQ_FLOOR, ACQ_REL, check_acq, check_mean, check_var, host_problem,
                       oracle_fit)
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def sample_indices(N, k_idx, runs=4, run_len=96, seed=0):
    rng = np.random.default_rng(seed)
    starts = [0, max(0, N - run_len)] + list(rng.integers(0, max(1, N - run_len), runs))
    idx = set(int(i) for i in k_idx)
    for s in starts:
        idx.update(range(int(s), min(N, int(s) + run_len)))
    return np.array(sorted(idx))


@pytest.mark.parametrize("wi", range(len(wl.WORKLOADS)), ids=[w.name for w in wl.WORKLOADS])
def test_full_size_workload(wi):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = wl.WORKLOADS[wi]
    hp = host_problem(w, threads=16)
    dev = torch.device("cuda")
    t = lambda a, dt: None if a is None else torch.as_tensor(a, dtype=dt, device=dev)
    f64, f32 = torch.float64, torch.float32
    mode = bt.BOUTE_ACQ_MC_HVI if w.mode == "mc" else bt.BOUTE_ACQ_EHVI2D
    e = bt.Engine(w.B, w.n, w.d, w.m, w.N, mode, w.S, w.k)
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device=dev)
    val = torch.empty((w.B, w.k), dtype=f32, device=dev)
    bt.boute_engine_step(e, t(hp.X, f64), t(hp.Y, f64), t(hp.ls, f64), t(hp.s2, f64),
                         t(hp.noise, f64), t(hp.ref, f64), t(hp.Xc, f32), t(hp.eps, f32), idx, val)
    acq = torch.empty((w.B, w.N), dtype=f32, device=dev)
    mean = torch.empty((w.B, w.m, w.N), dtype=f32, device=dev)
    var = torch.empty_like(mean)
    bt.boute_engine_scores(e, acq, mean, var)
    torch.cuda.synchronize()
    e.free()
    # top-k by properties: sorted, values are the scores at the indices, and
    # no unselected candidate scores above the k-th value
    kth = val[:, -1:]
    assert torch.all(val[:, :-1] >= val[:, 1:])
    assert torch.equal(torch.gather(acq, 1, idx), val)
    assert torch.all((acq > kth).sum(1) <= w.k - 1)
    assert torch.all((acq >= kth).sum(1) >= w.k)
    problems = [0] if w.B == 1 else [0, w.B // 2, w.B - 1]
    A, M, V, I = acq.cpu().numpy(), mean.cpu().numpy(), var.cpu().numpy(), idx.cpu().numpy()
    errs = {"mean": 0.0, "var": 0.0, "acq": 0.0}
    for b in problems:
        fp = oracle_fit(hp, b)
        sel = sample_indices(w.N, I[b], seed=b)
        mo, vo = opl.posterior(fp, hp.Xc[b][sel])
        for tt in range(w.m):
            errs["mean"] = max(errs["mean"], check_mean(M[b, tt, sel], mo[:, tt], fp.s2[tt]))
            errs["var"] = max(errs["var"], check_var(V[b, tt, sel], vo[:, tt], fp.s2[tt]))
        ao = opl.acquisition(fp, mo, vo, w.mode, None if hp.eps is None else hp.eps[b][sel])
        errs["acq"] = max(errs["acq"], check_acq(A[b, sel], ao))
        check_topk_against_oracle(hp, fp, w, b, A[b], I[b])
    # the measured errors (pytest -s shows them): mean relative to max(|mu|, s),
    # variance relative to s2, acquisition relative to max(|a|, 1e-3 max|a|)
    print(f"\n{w.name}: max err mean {errs['mean']:.2e} var {errs['var']:.2e} acq {errs['acq']:.2e}")


BAND = 4      # candidates within BAND tolerances below the GPU's k-th compete
MAX_BAND = 20000


def check_topk_against_oracle(hp, fp, w, b, acq, idx):
    """The oracle's top-k over the competing candidates equals the GPU's,
    except where the oracle's values are within tolerance of its k-th."""
    kth = float(acq[idx[-1]])
    tol = 2 * ACQ_REL * max(abs(kth), ACQ_FLOOR * float(np.abs(acq).max()))
    band = np.nonzero(acq >= kth - BAND * tol)[0]
    truncated = band.size > MAX_BAND
    if truncated:  # many near-equal scores: the strongest MAX_BAND by the GPU's values
        band = band[np.argsort(-acq[band], kind="stable")[:MAX_BAND]]
    cand = np.union1d(band, idx)
    mo, vo = opl.posterior(fp, hp.Xc[b][cand])
    ao = opl.acquisition(fp, mo, vo, w.mode, None if hp.eps is None else hp.eps[b][cand])
    order = np.argsort(-ao, kind="stable")
    okth = float(ao[order[w.k - 1]])
    mine = set(int(i) for i in idx)
    theirs = set(int(i) for i in cand[order[:w.k]])
    pos = {int(c): i for i, c in enumerate(cand)}
    for j in mine ^ theirs:
        assert abs(ao[pos[j]] - okth) <= tol, (
            f"problem {b}: candidate {j} {'selected' if j in mine else 'missed'} with oracle "
            f"value {ao[pos[j]]:.6g}, oracle k-th {okth:.6g}, tolerance {tol:.3g}")
    return truncated

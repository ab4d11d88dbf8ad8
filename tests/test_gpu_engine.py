"""The whole scoring step through the engine entry points: device inputs,
host inputs (copies inside the call, overlapped with the fit), graph replay
on a side stream, eager execution on the legacy default stream and the
stage-timing mode must all give the same selection, value for value, and the
same per-candidate scores as the step-by-step calls checked against the
oracle elsewhere. Consecutive host-input steps with different inputs catch
reuse of the engine's input buffers before the previous step is done."""
import dataclasses

import numpy as np
import pytest

from _pipeline import check_acq_end_to_end, gpu_pipeline, host_problem, oracle_fit
from oracle import pipeline as opl
from paper_2602_10729_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

CASES = [(0, 4096 + 77, 1), (1, 3000 + 5, 1), (4, 1500 + 1, 3)]


def _dev(hp):
    import torch
    t = lambda a, dt: None if a is None else torch.as_tensor(np.ascontiguousarray(a), dtype=dt,
                                                             device="cuda")
    f64, f32 = torch.float64, torch.float32
    return (t(hp.X, f64), t(hp.Y, f64), t(hp.ls, f64), t(hp.s2, f64), t(hp.noise, f64),
            t(hp.ref, f64), t(hp.Xc, f32), t(hp.eps, f32))


def _host(hp):
    import torch
    t = lambda a, dt: None if a is None else torch.as_tensor(np.ascontiguousarray(a),
                                                             dtype=dt).pin_memory()
    f64, f32 = torch.float64, torch.float32
    return (t(hp.X, f64), t(hp.Y, f64), t(hp.ls, f64), t(hp.s2, f64), t(hp.noise, f64),
            t(hp.ref, f64), t(hp.Xc, f32), t(hp.eps, f32))


def _engine(w):
    from paper_2602_10729_gb300 import boute as bt
    mode = bt.BOUTE_ACQ_MC_HVI if w.mode == "mc" else bt.BOUTE_ACQ_EHVI2D
    return bt.Engine(w.B, w.n, w.d, w.m, w.N, mode, w.S, w.k)


def _run(e, w, inputs, how):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    if how == "host":
        idx = torch.empty((w.B, w.k), dtype=torch.int64).pin_memory()
        val = torch.empty((w.B, w.k), dtype=torch.float32).pin_memory()
        bt.boute_engine_step_host(e, *inputs, idx, val)
        return idx.numpy().copy(), val.numpy().copy()
    idx = torch.empty((w.B, w.k), dtype=torch.int64, device="cuda")
    val = torch.empty((w.B, w.k), dtype=torch.float32, device="cuda")
    if how == "legacy":  # eager launches on the legacy default stream
        torch.cuda.synchronize()
        bt.boute_engine_step(e, *inputs, idx, val, stream=0)
    else:
        bt.boute_engine_step(e, *inputs, idx, val)
    return idx.cpu().numpy(), val.cpu().numpy()


@pytest.mark.parametrize("case", CASES, ids=lambda c: wl.WORKLOADS[c[0]].name)
def test_engine_paths_agree_and_match_oracle(case):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    wi, N, B = case
    w = wl.scaled(wl.WORKLOADS[wi], N=N, B=B)
    hp = host_problem(w)
    e = _engine(w)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        ref_idx, ref_val = _run(e, w, _dev(hp), "device")
        for how in ("device", "host", "legacy"):  # graph replay, host copies, eager
            idx, val = _run(e, w, _host(hp) if how == "host" else _dev(hp), how)
            assert np.array_equal(idx, ref_idx), how
            assert np.array_equal(val, ref_val), how
        bt.boute_engine_set_timing(e, True)
        idx, val = _run(e, w, _dev(hp), "device")
        times = bt.boute_engine_stage_times(e)
        assert np.array_equal(idx, ref_idx) and np.array_equal(val, ref_val)
        assert all(v > 0 for v in times.values()), times
        # live timing: the normal schedule with events on the step's stream
        bt.boute_engine_set_timing(e, bt.TIMING_LIVE)
        idx, val = _run(e, w, _dev(hp), "device")
        live = bt.boute_engine_stage_times(e)
        bt.boute_engine_set_timing(e, False)
        assert np.array_equal(idx, ref_idx) and np.array_equal(val, ref_val)
        assert live["front"] == 0 and live["fit"] > 0 and live["posterior"] > 0, live
        assert live["acquisition"] > 0 and live["topk"] >= 0, live
        acq = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
        bt.boute_engine_scores(e, acq=acq)
        torch.cuda.synchronize()
    e.free()
    A = acq.cpu().numpy()
    g = gpu_pipeline(hp)  # the step-by-step calls: same scores as the engine
    assert np.array_equal(g["acq"], A)
    for b in range(w.B):
        fp = oracle_fit(hp, b)
        mean, var = opl.posterior(fp, hp.Xc[b])
        eps = None if hp.eps is None else hp.eps[b]
        check_acq_end_to_end(A[b], lambda mm, vv: opl.acquisition(fp, mm, vv, w.mode, eps),
                             g["mean"][b].T, g["var"][b].T, mean, var, fp.s2)
        assert np.array_equal(ref_val[b], A[b][ref_idx[b]])


def test_consecutive_host_steps_with_new_inputs():
    w = wl.scaled(wl.WORKLOADS[1], N=2000 + 7, B=1)
    hp1 = host_problem(w)
    hp2 = host_problem(wl.scaled(w, N=w.N), threads=4)
    rng = np.random.default_rng(5)
    hp2.Xc[:] = rng.random(hp2.Xc.shape).astype(np.float32)
    hp2.eps[:] = rng.standard_normal(hp2.eps.shape).astype(np.float32)
    e = _engine(w)
    want = [_run(e, w, _dev(h), "device") for h in (hp1, hp2)]
    got = [_run(e, w, _host(h), "host") for h in (hp1, hp2, hp1)]
    e.free()
    for (gi, gv), (wi_, wv) in zip(got, want + want[:1]):
        assert np.array_equal(gi, wi_)
        assert np.array_equal(gv, wv)


# 2-objective Monte-Carlo steps with k <= 32 select inside the acquisition
# kernel; the stage-timing mode runs the separate selection launch instead.
# (B, N, S, k): the vectorised S = 128 path with many blocks per problem,
# the general S path, several problems, k = 1 and a ragged N.
FUSED = [(1, 65536 + 3, 128, 32), (3, 20000 + 11, 100, 17), (2, 5000, 128, 1), (1, 97, 33, 32)]


@pytest.mark.parametrize("B,N,S,k", FUSED)
def test_selection_in_acquisition_kernel_matches_separate_selection(B, N, S, k):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    base = wl.WORKLOADS[1]
    w = dataclasses.replace(wl.scaled(base, N=N, n=64, S=S), B=B, k=k,
                            seeds=tuple(range(1, B + 1)))
    hp = host_problem(w)
    e = _engine(w)
    got = [_run(e, w, _dev(hp), "device") for _ in range(3)]  # counters reset each step
    bt.boute_engine_set_timing(e, True)
    want = _run(e, w, _dev(hp), "device")  # eager on the legacy stream: plain event records
    assert all(v > 0 for v in bt.boute_engine_stage_times(e).values())
    acq = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
    bt.boute_engine_scores(e, acq=acq)
    torch.cuda.synchronize()
    e.free()
    A = acq.cpu().numpy()
    for gi, gv in got:
        assert np.array_equal(gi, want[0])
        assert np.array_equal(gv, want[1])
    for b in range(w.B):  # values descending, ties by index
        order = np.lexsort((np.arange(w.N), -A[b]))[:k]
        assert want[0][b].tolist() == order.tolist()


# Graph replay computes K* on a second stream beside the fit and the posterior
# only contracts it; stage-timing mode builds K* inside the posterior. Mean,
# variance, scores and selection must agree bit for bit. (workload, n, N, B):
# a ragged last chunk of training points, several problems, both
# acquisition modes, more than 256 training points.
TWO_PHASE = [(1, 77, 3000 + 5, 1), (4, 100, 1500 + 1, 3), (0, 32, 4096 + 77, 2),
             (1, 300, 700 + 3, 1), (4, 288, 500, 2)]  # (two column passes, split reduction)


@pytest.mark.parametrize("wi,n,N,B", TWO_PHASE)
def test_posterior_from_precomputed_kstar_matches_fused(wi, n, N, B):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    base = wl.WORKLOADS[wi]
    w = dataclasses.replace(wl.scaled(base, N=N, n=n), B=B, seeds=tuple(range(11, 11 + B)))
    hp = host_problem(w)
    e = _engine(w)
    out = []
    for timing in (False, True, bt.TIMING_LIVE):
        bt.boute_engine_set_timing(e, timing)
        idx, val = _run(e, w, _dev(hp), "device")
        mean = torch.empty((w.B, w.m, w.N), dtype=torch.float32, device="cuda")
        var = torch.empty_like(mean)
        acq = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
        bt.boute_engine_scores(e, acq=acq, mean=mean, var=var)
        torch.cuda.synchronize()
        out.append((idx, val, acq.cpu().numpy(), mean.cpu().numpy(), var.cpu().numpy()))
    e.free()
    for other in out[1:]:
        for a, b in zip(out[0], other):
            assert np.array_equal(a, b)


# Pipelined host-input steps: consecutive calls alternate between two device
# input sets and overlap one step's copies with the previous step's
# computation; each step's results must equal the device-input step's.
@pytest.mark.parametrize("wi,N,B", [(1, 2000 + 7, 1), (4, 1500 + 1, 3)])
def test_pipelined_host_steps_match_device_steps(wi, N, B):
    import torch

    from paper_2602_10729_gb300 import boute as bt
    w = wl.scaled(wl.WORKLOADS[wi], N=N, B=B)
    hp1 = host_problem(w)
    hp2 = host_problem(wl.scaled(w, N=w.N), threads=4)
    rng = np.random.default_rng(11)
    hp2.Xc[:] = rng.random(hp2.Xc.shape).astype(np.float32)
    if hp2.eps is not None:
        hp2.eps[:] = rng.standard_normal(hp2.eps.shape).astype(np.float32)
    e = _engine(w)
    want = [_run(e, w, _dev(h), "device") for h in (hp1, hp2)]
    inputs = [_host(h) for h in (hp1, hp2, hp1, hp2, hp1)]
    outs = [(torch.empty((w.B, w.k), dtype=torch.int64).pin_memory(),
             torch.empty((w.B, w.k), dtype=torch.float32).pin_memory()) for _ in inputs]
    for inp, (i, v) in zip(inputs, outs):
        bt.boute_engine_step_host_async(e, *inp, i, v)
    bt.boute_engine_sync(e)
    e.free()
    for (i, v), (wi_, wv) in zip(outs, want + want + want[:1]):
        assert np.array_equal(i.numpy(), wi_)
        assert np.array_equal(v.numpy(), wv)


# (workload, cap, sizes): the engine is created for `cap` observations and
# then stepped at each size in turn, on a stream (graphs re-captured per size),
# from host buffers and eagerly; sizes above 512 use the posterior's K* cache, 2-objective
# Monte-Carlo steps the in-kernel selection whose scratch depends on n
SET_N_CASES = [(0, 300, [300, 37, 129, 200]), (1, 160, [64, 160, 95]),
               (3, 1024, [1024, 700, 513, 600])]


@pytest.mark.parametrize("case", SET_N_CASES, ids=lambda c: wl.WORKLOADS[c[0]].name)
def test_engine_set_n_matches_fresh_engine(case):
    """A capacity-sized engine re-planned to a smaller n gives the same
    selection, bit for bit, as an engine created for that n."""
    import torch

    from paper_2602_10729_gb300 import boute as bt
    wi, cap, sizes = case
    base = wl.WORKLOADS[wi]
    e = _engine(wl.scaled(base, N=2048 + 33, B=1, n=cap))
    stream = torch.cuda.Stream()
    for n in sizes:
        w = wl.scaled(base, N=2048 + 33, B=1, n=n)
        hp = host_problem(w)
        bt.boute_engine_set_n(e, n)
        fresh = _engine(w)
        with torch.cuda.stream(stream):
            ref_idx, ref_val = _run(fresh, w, _dev(hp), "device")
            for how in ("device", "device", "host", "legacy"):  # capture, replay, ...
                idx, val = _run(e, w, _host(hp) if how == "host" else _dev(hp), how)
                assert np.array_equal(idx, ref_idx), (n, how)
                assert np.array_equal(val, ref_val), (n, how)
        fresh.free()
    with pytest.raises(RuntimeError):
        bt.boute_engine_set_n(e, cap + 1)
    with pytest.raises(RuntimeError):
        bt.boute_engine_set_n(e, 0)
    e.free()

"""The bounds-checked debug build (BOUTE_DEBUG_BOUNDS): every path of the
library runs on small and ragged cases with the index checks compiled in
(bulk-copy ranges, operand images, outputs, strips and boxes, selection), and
no index may fall outside its extent. The debug library is loaded in a child
process so that this process keeps the product library; the product library
answers the report call with BOUTE_ERR_UNSUPPORTED."""
import os
import subprocess
import sys
import textwrap

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

CHILD = textwrap.dedent(r"""
    import dataclasses, sys
    sys.path.insert(0, ROOT); sys.path.insert(0, HERE)
    import numpy as np
    from paper_2602_10729_gb300 import boute as bt, build as bld, workloads as wl
    bt.load(bld.build(debug=True))
    import torch
    from _pipeline import gpu_pipeline, host_problem
    import test_gpu_noisy as tn

    def report(what):
        r = bt.boute_bounds_report()
        print(what, "ok" if r is None else f"VIOLATION unit={r[0]} line={r[1]} index={r[2]} extent={r[3]}")
        return r is None

    ok = True
    # the step one entry point at a time: every workload, ragged tiles, the
    # composite kernel, a constrained acquisition
    for wi, N, B, n in [(0, 4096 + 77, 1, 32), (1, 3000 + 5, 1, 128), (2, 2000 + 3, 1, 512),
                        (3, 700 + 11, 1, 1024), (4, 1500 + 1, 3, 256), (1, 999, 1, 37),
                        (2, 1500 + 7, 1, 600)]:
        w = wl.scaled(wl.WORKLOADS[wi], N=N, B=B, n=n)
        hp = host_problem(w)
        g = gpu_pipeline(hp)
        assert g["status"] == 0, g["status"]
        ok &= report(f"pipeline {w.name} n={n}")
    w = wl.scaled(wl.composite(wl.WORKLOADS[1]), N=1500 + 3, B=1)
    gpu_pipeline(host_problem(w))
    ok &= report("composite kernel")
    w = wl.scaled(wl.WORKLOADS[1], N=2000 + 9, B=1)
    gpu_pipeline(host_problem(w), cons=np.tile([0.3, 0.5], (1, 1)))
    ok &= report("constrained")
    # the noisy acquisition
    for case in tn.CASES:
        wi, N, n, S, B, constrained = case
        w = tn._workload(wi, N, n, S, B)
        hp = host_problem(w)
        z = np.stack([wl.insample_normals(w, b) for b in range(B)])
        tn._gpu(hp, z, tn._cons(hp) if constrained else None)
        ok &= report(f"noisy {case}")
    # engine steps (graph with K* beside the fit, fused selection, host inputs)
    for wi, N, mode in [(1, 4096 + 3, bt.BOUTE_ACQ_MC_HVI), (0, 2048 + 1, bt.BOUTE_ACQ_EHVI2D),
                        (1, 2048 + 5, bt.BOUTE_ACQ_NEHVI)]:
        w = wl.scaled(wl.WORKLOADS[wi], N=N, B=1)
        if mode == bt.BOUTE_ACQ_NEHVI:
            w = dataclasses.replace(w, mode="mc", S=64)
        hp = host_problem(w)
        e = bt.Engine(1, w.n, w.d, w.m, N, mode, w.S, w.k)
        inputs = tn._engine_inputs(hp) if mode != bt.BOUTE_ACQ_EHVI2D else tn._engine_inputs(
            dataclasses.replace(hp, eps=np.zeros((1, 1, 1, 1), np.float32)))
        if mode == bt.BOUTE_ACQ_EHVI2D:
            inputs = inputs[:-1] + (None,)
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            for how in ("device", "device", "host", "legacy"):
                if how == "host" and mode == bt.BOUTE_ACQ_EHVI2D:
                    continue
                tn._engine_step(e, w, inputs, how)
        e.free()
        ok &= report(f"engine mode {mode}")
    print("ALL_CLEAN" if ok else "FOUND_VIOLATIONS")
""")


def test_no_index_outside_its_extent():
    env = dict(os.environ)
    code = f"ROOT = {ROOT!r}\nHERE = {HERE!r}\n" + CHILD
    res = subprocess.run([sys.executable, "-c", code], cwd=HERE, env=env, capture_output=True,
                         text=True, timeout=1500)
    out = res.stdout + res.stderr
    assert res.returncode == 0, out[-4000:]
    print(res.stdout)
    assert "ALL_CLEAN" in res.stdout, res.stdout[-4000:]
    assert res.stdout.count(" ok") >= 16  # every path above reported


def test_product_library_has_no_checks():
    from paper_2602_10729_gb300 import boute as bt
    with pytest.raises(bt.BouteError) as ei:
        bt.boute_bounds_report()
    assert ei.value.code == bt.BOUTE_ERR_UNSUPPORTED

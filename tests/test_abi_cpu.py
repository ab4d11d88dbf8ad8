"""Host-side checks of the C-ABI library (no GPU needed): it builds for
sm_103a, loads, exports every entry point that include/boute.h declares,
and rejects bad arguments before touching a device."""
import ctypes
import os
import re

import pytest

from paper_2602_10729_gb300 import boute as bt
from paper_2602_10729_gb300 import build as bld

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    bld.build()
    return bt.load()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "boute.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(boute_\w+)\s*\(", src)))


def test_header_declares_the_binding_surface():
    assert declared_functions() == sorted(bt.SYMBOLS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_library_targets_sm103a_only():
    out = os.popen(f"/usr/local/cuda/bin/cuobjdump --list-elf {bld.LIB} 2>/dev/null").read()
    archs = set(re.findall(r"sm_\d+a?", out))
    assert archs == {"sm_103a"}, archs


def test_status_strings(lib):
    assert bt.status_string(0) == "ok"
    assert "positive definite" in bt.status_string(2)
    assert bt.status_string(99) == "unknown status"


def test_invalid_arguments_are_rejected_before_any_device_call(lib):
    h = ctypes.c_void_p()
    assert lib.boute_gp_create(0, 4, 2, 1, ctypes.byref(h)) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_create(1, 4, 33, 1, ctypes.byref(h)) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_create(1, 4096, 2, 1, ctypes.byref(h)) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_create(1, 4, 2, 1, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_select_topk(None, 1, 10, 3, None, None, None) == bt.BOUTE_ERR_INVALID_ARG
    p = ctypes.c_void_p(16)
    assert lib.boute_select_topk(p, 1, 10, 11, p, p, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_select_topk(p, 1, 10, 0, p, p, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_engine_create(1, 8, 2, 3, 100, bt.BOUTE_ACQ_EHVI2D, 0, 4,
                                   ctypes.byref(h)) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_acq_mc_hvi(p, p, 1, 10, 4, p, p, p, 4, p, 8, 32, None, p, None) in (
        bt.BOUTE_ERR_UNSUPPORTED, bt.BOUTE_ERR_INVALID_ARG)
    assert lib.boute_engine_set_constraints(None, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_status(None, None) == bt.BOUTE_ERR_INVALID_ARG
    # outcome transforms: unknown codes (3: both log and logit; 8: no such bit)
    for codes in ([3, 0], [0, 8], [-1, 0]):
        arr = (ctypes.c_int * 2)(*codes)
        assert lib.boute_standardize(p, 1, 4, 2, arr, p, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_engine_set_outcome_transforms(None, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_selftest_wait(0, 3_000_000_000, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_engine_set_kernel(None, 0, None) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_set_kernel(None, 0, None) == bt.BOUTE_ERR_INVALID_ARG
    # precision tiers
    assert lib.boute_gp_set_precision(None, bt.BOUTE_PREC_FP64) == bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_posterior_fp64(None, p, 10, p, p, None) == bt.BOUTE_ERR_INVALID_ARG
    # hyperparameter learning: restarts, steps, step size, d_tau
    assert lib.boute_gp_learn(p, p, 1, 8, 2, 2, p, 0, 5, 0.1, p, p, None, None) == \
        bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_learn(p, p, 1, 8, 2, 2, p, 1, -1, 0.1, p, p, None, None) == \
        bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_learn(p, p, 1, 8, 2, 2, p, 1, 5, float("nan"), p, p, None, None) == \
        bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_learn_k(p, p, 1, 8, 2, 2, 3, p, p, 1, 5, 0.1, p, p, None, None) == \
        bt.BOUTE_ERR_INVALID_ARG
    assert lib.boute_gp_learn_k(p, p, 1, 8, 2, 2, 1, None, p, 1, 5, 0.1, p, p, None, None) == \
        bt.BOUTE_ERR_INVALID_ARG
    # the loop: no configuration, a budget below the initial observations
    n_out, conv = ctypes.c_int(), ctypes.c_int()
    fn = bt.ObjectiveFn(lambda *a: 0)
    assert lib.boute_mobo_run(None, 2, 2, p, 10, None, p, None, None, 0, None, p, p, p, p, p, 4,
                              fn, None, p, None, ctypes.byref(n_out),
                              ctypes.byref(conv)) == bt.BOUTE_ERR_INVALID_ARG
    cfg = bt.MoboConfig(bt.BOUTE_ACQ_EHVI2D, 0, 3, 5, 0, 0.05, 0)
    assert lib.boute_mobo_run(ctypes.byref(cfg), 2, 2, p, 10, None, p, None, None, 0, None, p, p,
                              p, p, p, 4, fn, None, p, None, ctypes.byref(n_out),
                              ctypes.byref(conv)) == bt.BOUTE_ERR_INVALID_ARG
    cfg = bt.MoboConfig(bt.BOUTE_ACQ_MC_HVI, 0, 8, 5, 0, 0.05, 0)  # MC without samples
    assert lib.boute_mobo_run(ctypes.byref(cfg), 2, 2, p, 10, None, p, None, None, 0, None, p, p,
                              p, p, p, 4, fn, None, p, None, ctypes.byref(n_out),
                              ctypes.byref(conv)) == bt.BOUTE_ERR_INVALID_ARG


def test_valid_calls_without_a_device_report_unsupported(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a device is present")
    h = ctypes.c_void_p()
    assert lib.boute_gp_create(1, 4, 2, 1, ctypes.byref(h)) == bt.BOUTE_ERR_UNSUPPORTED
    assert not h.value

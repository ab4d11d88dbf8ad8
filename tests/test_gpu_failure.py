"""Failure detection without a GPU fault: every device-side wait of the
library is bounded and reports BOUTE_ERR_TIMEOUT when its bound runs out.
The self-test entry point runs one such wait, through the same bounded-wait
helper the kernels use, on an mbarrier that nothing arrives on (with a short
bound), and the device must stay usable afterwards."""
import time

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_the_device_stays_usable():
    import torch

    from paper_2602_10729_gb300 import boute as bt
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    st = bt.boute_selftest_wait(False, 3_000_000)  # 3 ms, nothing arrives
    dt = time.perf_counter() - t0
    assert st == bt.BOUTE_ERR_TIMEOUT
    assert dt >= 0.003
    assert bt.boute_selftest_wait(True, 3_000_000) == bt.BOUTE_OK  # the arrival completes it
    # the context is intact: library and PyTorch work as before
    v = torch.arange(1000, dtype=torch.float32, device="cuda")[None].contiguous()
    idx = torch.empty((1, 3), dtype=torch.int64, device="cuda")
    val = torch.empty((1, 3), dtype=torch.float32, device="cuda")
    bt.boute_select_topk(v, 1, 1000, 3, idx, val)
    assert idx.cpu().numpy().tolist() == [[999, 998, 997]]
    assert np.allclose(val.cpu().numpy(), [[999, 998, 997]])

"""boute_select_topk_noalloc, the selection whose scratch is a fixed array
compiled into the library: called twice in a row through the C-ABI, it must
return what boute_select_topk returns, index for index and value for value,
up to the largest request its array holds; a larger request is refused before
anything is launched. Collected last so it also runs after every other test
has used the library (and the CUDA memory pool) in the same process."""
import numpy as np
import pytest

from paper_2602_10729_gb300 import boute as bt

pytestmark = pytest.mark.gpu

# (B, N, k): one segment, two levels, a ragged last segment, several problems,
# the largest k, and a request that fills the array exactly
CASES = [(1, 1000, 10), (1, 2048, 64), (2, 70_001, 64), (3, 300_000, 1024), (1, 1, 1),
         (4, 1 << 22, 64), (3, 700_001, 17)]


def _scratch_bytes(B, N, k):
    nseg = -(-N // 2048)
    return 0 if nseg <= 1 else 2 * B * nseg * max(k, 32) * 8


@pytest.mark.parametrize("B,N,k", CASES)
def test_noalloc_matches_pool_scratch_twice(B, N, k):
    import torch
    assert _scratch_bytes(B, N, k) <= bt.TOPK_NOALLOC_SCRATCH_BYTES
    g = torch.Generator(device="cpu").manual_seed(B * 1_000_003 + N + k)
    vals = torch.rand((B, N), generator=g, dtype=torch.float32)
    vals = torch.round(vals * 4096) / 4096  # plenty of ties
    a = vals.to("cuda")
    want_i = torch.empty((B, k), dtype=torch.int64, device="cuda")
    want_v = torch.empty((B, k), dtype=torch.float32, device="cuda")
    bt.boute_select_topk(a, B, N, k, want_i, want_v)
    for _ in range(2):
        idx = torch.full((B, k), -1, dtype=torch.int64, device="cuda")
        val = torch.full((B, k), float("nan"), dtype=torch.float32, device="cuda")
        bt.boute_select_topk_noalloc(a, B, N, k, idx, val)
        torch.cuda.synchronize()
        assert torch.equal(idx, want_i)
        assert torch.equal(val, want_v)
    # and the selection is the right one: values descending, ties by index
    iv = want_i.cpu().numpy()
    vv = vals.numpy()
    for b in range(B):
        order = np.lexsort((np.arange(N), -vv[b]))[:k]
        assert iv[b].tolist() == order.tolist()


def test_noalloc_refuses_requests_beyond_its_array():
    import torch
    B, N, k = 5, 1 << 22, 64  # 10 MiB of scratch: above the 8 MiB array
    assert _scratch_bytes(B, N, k) > bt.TOPK_NOALLOC_SCRATCH_BYTES
    a = torch.zeros((B, N), dtype=torch.float32, device="cuda")
    idx = torch.empty((B, k), dtype=torch.int64, device="cuda")
    val = torch.empty((B, k), dtype=torch.float32, device="cuda")
    before = bt.boute_launch_count()
    with pytest.raises(bt.BouteError) as e:
        bt.boute_select_topk_noalloc(a, B, N, k, idx, val)
    assert e.value.code == bt.BOUTE_ERR_UNSUPPORTED
    assert bt.boute_launch_count() == before

"""The bounded-wait path on the GPU: a wait that nothing completes gives up
after its limit, is reported by hill_sync_status as HILL_ERR_TIMEOUT, and
leaves the context usable (a normal call right after it succeeds).  No fault,
trap or unbounded spin is involved."""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2602_18750_gb300 import build, hill
    build.build()
    hill.load()
    return hill


def test_wait_times_out_and_context_survives(H):
    H.hill_sync_status()                       # start from a clean error word
    t0 = time.time()
    H.hill_selftest_wait(20000)                # 20 ms
    with pytest.raises(H.HillError) as e:
        H.hill_sync_status()
    assert e.value.status == H.HILL_ERR_TIMEOUT
    assert time.time() - t0 >= 0.015           # it really waited for its limit
    H.hill_sync_status()                       # the word was cleared
    # the context still runs kernels: a small selection
    s = torch.randn(2, 300, device="cuda")
    q = torch.zeros(2, 4, 128, dtype=torch.float16, device="cuda")
    K = torch.zeros(2, 4, 300, 128, dtype=torch.float16, device="cuda")
    desc = H.make_desc(q, K)
    idx = torch.empty(2, 30, dtype=torch.int32, device="cuda")
    cnt = torch.empty(2, dtype=torch.int32, device="cuda")
    lens = torch.tensor([300, 120], dtype=torch.int32, device="cuda")
    k = torch.tensor([30, 12], dtype=torch.int32, device="cuda")
    H.hill_topk_select(desc, s, lens, k, 30, idx, cnt)
    H.hill_sync_status()
    assert cnt.tolist() == [30, 12]

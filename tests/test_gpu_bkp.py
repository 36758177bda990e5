"""GPU parity of the BKP bookkeeping (Sec. 4.2): pinned recent window, ranked
older tokens and the saturating hit-rate table, through the C ABI, against
the CPU oracle (oracle.bkp_select) on the same keys.  Index sets, counts and
hit tables are compared exactly: the keys are float32 values that the oracle
ranks exactly in float64.
"""
import numpy as np
import pytest
import torch

from paper_2602_18750_gb300 import inputs
from parity_util import check_attn, check_scores

pytestmark = pytest.mark.gpu

ATTN, RAW = 0, 1


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2602_18750_gb300 import build, hill
    build.build()
    hill.load()
    return hill


def _desc(H, B, cap):
    q = torch.zeros(B, 4, 128, dtype=torch.float16, device="cuda")
    K = torch.zeros(B, 4, 8, 128, dtype=torch.float16, device="cuda")
    d = H.make_desc(q, K)
    d.capacity = cap
    return d


def _i32(x):
    return torch.tensor(x, dtype=torch.int32, device="cuda")


@pytest.mark.parametrize("cap", [5000, 40000, 131072 + 7])
@pytest.mark.parametrize("recent", [0, 37, 4000])
def test_bkp_select_matches_oracle_over_steps(H, oracle_mod, cap, recent):
    """Single-CTA and 4- and 8-CTA cluster selections, three decode steps with
    the hit table carried from step to step; heavy exact ties in step 0."""
    B = 3
    g = torch.Generator().manual_seed(cap + recent)
    lens = [cap, cap // 2 + 3, min(cap, 3 * recent + 11)]
    k = [cap // 10, 2048, 100]
    max_k = max(k) + recent
    desc = _desc(H, B, cap)
    hits = torch.zeros(B, cap, dtype=torch.int16, device="cuda")
    hits_o = np.zeros((B, cap), dtype=np.uint16)
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    for step in range(3):
        s = torch.rand(B, cap, generator=g) ** 4
        if step == 0:
            s = torch.round(s * 8) / 8
        H.hill_topk_select_bkp(desc, s.cuda(), _i32(lens), _i32(k), recent, max_k, idx, cnt, hits)
        H.hill_sync_status()
        idx_o, cnt_o, rc, hits_o = oracle_mod.bkp_select(s.numpy().astype(np.float64), lens, k, recent,
                                                         max_k, hits_o)
        assert rc == 0
        assert np.array_equal(cnt.cpu().numpy(), cnt_o)
        assert np.array_equal(idx.cpu().numpy(), idx_o)
        assert np.array_equal(hits.cpu().numpy().view(np.uint16), hits_o)


def test_bkp_window_wider_than_budget(H, oracle_mod):
    """A window wider than max_k keeps its most recent tokens and is reported
    as a device-side budget error (HILL_ERR_DEVICE)."""
    B, cap, max_k = 2, 900, 64
    s = torch.rand(B, cap, generator=torch.Generator().manual_seed(5))
    lens, k = [900, 500], [10, 30]
    desc = _desc(H, B, cap)
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_topk_select_bkp(desc, s.cuda(), _i32(lens), _i32(k), 100, max_k, idx, cnt)
    with pytest.raises(H.HillError) as e:
        H.hill_sync_status()
    assert e.value.status == H.HILL_ERR_DEVICE
    idx_o, cnt_o, rc, _ = oracle_mod.bkp_select(s.numpy().astype(np.float64), lens, k, 100, max_k)
    assert rc == 2
    assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)


def test_bkp_zero_window_equals_plain_select(H):
    B, cap = 2, 3000
    s = torch.randn(B, cap, generator=torch.Generator().manual_seed(6)).cuda()
    lens, k = _i32([3000, 1777]), _i32([300, 1777])
    desc = _desc(H, B, cap)
    a = [torch.empty(B, 1777, dtype=torch.int32, device="cuda") for _ in range(2)]
    c = [torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(2)]
    H.hill_topk_select(desc, s, lens, k, 1777, a[0], c[0])
    H.hill_topk_select_bkp(desc, s, lens, k, 0, 1777, a[1], c[1])
    H.hill_sync_status()
    assert torch.equal(a[0], a[1]) and torch.equal(c[0], c[1])


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("cap", [1500, 40000], ids=["single-kernel", "statistics-kernel"])
def test_evict_step_bkp(H, oracle_mod, mode, cap):
    """The fused step with BKP equals hill_score + hill_topk_select_bkp (the
    ATTN path starts its selection from a histogram that must leave the
    pinned window out), matches the oracle's scores and BKP selection, and
    its attention matches the oracle on the GPU's own index set."""
    B, Hq, Hkv, recent = 3, 8, 2, 64
    lens = [cap, cap * 3 // 5 + 1, 40]
    k = [cap // 10, cap // 17, 10]
    max_k = k[0] + recent
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=21)
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K, V)
    ws = H.alloc_workspace(desc, mode, max_k)
    k_t = _i32(k)
    scores = torch.zeros(B, cap, device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    hits = torch.zeros(B, cap, dtype=torch.int16, device="cuda")
    out = torch.empty(B, Hq, 128, device="cuda")
    H.hill_evict_step_bkp(desc, q, K, V, lens_t, k_t, recent, max_k, mode, None, scores, idx, cnt, hits, out, ws)
    s2 = torch.zeros(B, cap, device="cuda")
    idx2 = torch.empty_like(idx)
    cnt2 = torch.empty_like(cnt)
    hits2 = torch.zeros_like(hits)
    H.hill_score(desc, q, K, lens_t, mode, s2, ws=ws)
    H.hill_topk_select_bkp(desc, s2, lens_t, k_t, recent, max_k, idx2, cnt2, hits2)
    H.hill_sync_status()
    assert torch.equal(idx, idx2) and torch.equal(cnt, cnt2) and torch.equal(hits, hits2)
    z = oracle_mod.logits(q.cpu(), K.cpu(), lens)
    s_ref = oracle_mod.scores(mode, z, lens)
    check_scores(scores.cpu().numpy(), s_ref, lens)
    # selection: the oracle's BKP rule on the GPU's own float32 scores
    s_gpu = scores.cpu().numpy().astype(np.float64)
    idx_o, cnt_o, rc, hits_o = oracle_mod.bkp_select(s_gpu, lens, k, recent, max_k,
                                                     np.zeros((B, cap), np.uint16))
    assert rc == 0
    assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)
    assert np.array_equal(hits.cpu().numpy().view(np.uint16), hits_o)
    o_ref = oracle_mod.sparse_attn(q.cpu(), K.cpu(), V.cpu(), idx.cpu().numpy(), cnt.cpu().numpy())
    check_attn(out.cpu().numpy(), o_ref)

"""GPU parity of the per-KV-head selection (hill_evict_step_kvh): scores
aggregated over each KV head's query group, one top-k per (b, g), and the
attention of each query group over its KV head's own rows, against the
oracle's per-KV-head composition (oracle.scores_kvh / topk_kvh /
sparse_attn_kvh) on the same seeded inputs.
"""
import numpy as np
import pytest
import torch

from paper_2602_18750_gb300 import inputs
from parity_util import check_attn, check_scores, check_selection

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


def _i32(x):
    return torch.tensor(x, dtype=torch.int32, device="cuda")


SHAPES = [
    # B, H, Hkv, cap, lens, k
    (3, 8, 8, 700, [700, 333, 40], [140, 66, 40]),
    (2, 32, 8, 600, [600, 257], [120, 51]),
    (2, 8, 1, 300, [300, 299], [30, 299]),
    (4, 16, 2, 129, [129, 0, 64, 95], [13, 3, 64, 0]),
    (2, 32, 2, 400, [400, 177], [40, 17]),   # 16 query heads per KV head
    (2, 32, 1, 300, [300, 123], [30, 12]),   # MQA: one KV head, 32 query heads
    (2, 28, 4, 300, [300, 77], [30, 7]),     # 7 query heads per KV head
    (2, 12, 1, 200, [200, 64], [20, 6]),     # 12 = 8 + 4 heads on one KV head
    (1, 40, 40, 200, [200], [40]),           # 40 KV heads: two scoring passes
]


def _run(H, q, K, V, lens_t, k, max_k, mode, accum=None):
    B, Hq, _ = q.shape
    Hkv, cap = K.shape[1], K.shape[2]
    desc = H.make_desc(q, K, V)
    ws = H.alloc_workspace(desc, mode, max_k)
    # NaN-filled, so that a row read before any pass wrote it fails the check
    scores = torch.full((B, Hkv, cap), float("nan"), device="cuda")
    idx = torch.empty(B, Hkv, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, Hkv, dtype=torch.int32, device="cuda")
    out = torch.empty(B, Hq, 128, device="cuda")
    H.hill_evict_step_kvh(desc, q, K, V, lens_t, _i32(k), max_k, mode, accum, scores, idx, cnt, out, ws)
    H.hill_sync_status()
    return scores, idx, cnt, out


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_evict_step_kvh_matches_oracle(H, oracle_mod, mode, dtype, shape):
    B, Hq, Hkv, cap, lens, k = shape
    max_k = max(k) + 1
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=dtype, seed=cap + Hkv, kind="zipf")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    scores, idx, cnt, out = _run(H, q, K, V, lens_t, k, max_k, mode)
    z = oracle_mod.logits(q.cpu(), K.cpu(), lens)
    s_ref = oracle_mod.scores_kvh(mode, z, lens, Hkv)
    rows_lens = np.repeat(lens, Hkv).tolist()
    check_scores(scores.cpu().numpy().reshape(B * Hkv, cap), s_ref.reshape(B * Hkv, cap), rows_lens)
    check_selection(idx.cpu().numpy().reshape(B * Hkv, max_k), cnt.cpu().numpy().reshape(-1),
                    s_ref.reshape(B * Hkv, cap), rows_lens, np.repeat(k, Hkv), max_k)
    o_ref = oracle_mod.sparse_attn_kvh(q.cpu(), K.cpu(), V.cpu(), idx.cpu().numpy(), cnt.cpu().numpy())
    check_attn(out.cpu().numpy(), o_ref)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_kvh_accumulates_over_steps(H, oracle_mod, mode):
    B, Hq, Hkv, cap = 2, 16, 4, 400
    lens, k = [400, 211], [80, 42]
    accum = torch.zeros(B, Hkv, cap, device="cuda")
    acc_ref = np.zeros((B, Hkv, cap))
    for step in range(3):
        q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=50 + step)
        q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
        _, idx, cnt, _ = _run(H, q, K, V, lens_t, k, 80, mode, accum=accum)
        z = oracle_mod.logits(q.cpu(), K.cpu(), lens)
        s_ref = oracle_mod.scores_kvh(mode, z, lens, Hkv)
        for b in range(B):
            acc_ref[b, :, : lens[b]] += s_ref[b, :, : lens[b]]
    rows_lens = np.repeat(lens, Hkv).tolist()
    check_scores(accum.cpu().numpy().reshape(B * Hkv, cap), acc_ref.reshape(B * Hkv, cap), rows_lens,
                 what="accum")
    check_selection(idx.cpu().numpy().reshape(B * Hkv, 80), cnt.cpu().numpy().reshape(-1),
                    acc_ref.reshape(B * Hkv, cap), rows_lens, np.repeat(k, Hkv), 80)


def test_kvh_long_sequences_statistics_kernel(H, oracle_mod):
    """Per-KV-head sums on the two-kernel normalisation (sequences long
    enough for more than two normalisation CTAs per SM)."""
    B, Hq, Hkv, cap = 2, 16, 4, 40000
    lens, k = [40000, 31111], [3000, 1000]
    max_k = 3001
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.bfloat16, seed=77, kind="zipf")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    scores, idx, cnt, out = _run(H, q, K, V, lens_t, k, max_k, ATTN)
    z = oracle_mod.logits(q.cpu(), K.cpu(), lens)
    s_ref = oracle_mod.scores_kvh(ATTN, z, lens, Hkv)
    rows_lens = np.repeat(lens, Hkv).tolist()
    check_scores(scores.cpu().numpy().reshape(B * Hkv, cap), s_ref.reshape(B * Hkv, cap), rows_lens)
    check_selection(idx.cpu().numpy().reshape(B * Hkv, max_k), cnt.cpu().numpy().reshape(-1),
                    s_ref.reshape(B * Hkv, cap), rows_lens, np.repeat(k, Hkv), max_k)
    o_ref = oracle_mod.sparse_attn_kvh(q.cpu(), K.cpu(), V.cpu(), idx.cpu().numpy(), cnt.cpu().numpy())
    check_attn(out.cpu().numpy(), o_ref)


def test_kvh_with_one_kv_head_equals_sequence_step(H):
    """Hkv = 1: the per-KV-head step is the per-sequence step."""
    B, Hq, cap = 3, 8, 500
    lens, k = [500, 377, 90], [100, 75, 18]
    q, K, V, lens_t = inputs.random_case(B, Hq, 1, 128, cap, lens, dtype=torch.float16, seed=61, kind="zipf")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    for mode in (ATTN, RAW):
        scores, idx, cnt, out = _run(H, q, K, V, lens_t, k, 100, mode)
        ev = H.Evictor(q, K, V, 100, mode=mode)
        ev.step(q, K, V, lens_t, _i32(k))
        H.hill_sync_status()
        assert torch.equal(idx[:, 0], ev.idx) and torch.equal(cnt[:, 0], ev.count)
        assert torch.equal(out, ev.out)
        for b in range(B):
            assert torch.equal(scores[b, 0, : lens[b]], ev.scores[b, : lens[b]])

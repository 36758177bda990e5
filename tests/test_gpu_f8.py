"""GPU parity of the asymmetric-precision scoring (Sec. 4.4): the E4M3 key
shadow written by hill_quantize_k (bit-exact against the oracle's float32
quantisation), the scores of hill_score_f8 against the oracle's logits on the
8-bit operands, and hill_evict_step_f8 (selection from the shadow, attention
on the original 16-bit keys and values).  The small shapes take the
warp-level E4M3 kernel; TC_SHAPES (2 to 16 query heads per KV head, at least
64 MB of codes) take the tensor-core kernel, through hill_score_f8 and the
split step.
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


def _shadow(H, desc, K, lens):
    k8, ks = H.alloc_shadow(desc)
    B = desc.batch
    H.hill_quantize_k(desc, K, _i32([0] * B), _i32(lens), desc.capacity, k8, ks)
    return k8, ks


@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_quantize_k_bit_exact(H, oracle_mod, dtype):
    """Codes and scales of every row equal the oracle's; rows outside the
    requested ranges are left untouched; an all-zero row gives zeros."""
    B, Hkv, cap = 3, 4, 300
    g = torch.Generator().manual_seed(1)
    K = (torch.randn(B, Hkv, cap, 128, generator=g) * torch.logspace(-4, 3, cap)[None, None, :, None]).to(dtype)
    K[1, 2, 7] = 0
    K[2, 0, 9, :5] = -0.0
    Kd = K.cuda()
    q = torch.zeros(B, 4 * Hkv, 128, dtype=dtype, device="cuda")
    desc = H.make_desc(q, Kd)
    k8, ks = H.alloc_shadow(desc)
    k8.fill_(0xAB)
    ks.fill_(-1.0)
    begin, end = [0, 17, 250], [300, 200, 251]
    H.hill_quantize_k(desc, Kd, _i32(begin), _i32(end), 300, k8, ks)
    H.hill_sync_status()
    codes, scale = oracle_mod.quantize_rows(K)
    got_c, got_s = k8.cpu().numpy(), ks.cpu().numpy()
    for b in range(B):
        r = slice(begin[b], end[b])
        assert np.array_equal(got_c[b, :, r], codes[b, :, r])
        assert np.array_equal(got_s[b, :, r], scale[b, :, r])
        assert np.all(got_c[b, :, : begin[b]] == 0xAB) and np.all(got_c[b, :, end[b]:] == 0xAB)
        assert np.all(got_s[b, :, : begin[b]] == -1.0)


def test_quantize_k_token_major_layout(H, oracle_mod):
    """A token-major cache [B][cap][Hkv][d] quantises to the same dense shadow."""
    B, Hkv, cap = 2, 2, 97
    g = torch.Generator().manual_seed(2)
    Kt = torch.randn(B, cap, Hkv, 128, generator=g).half().cuda()
    K = Kt.permute(0, 2, 1, 3)                      # [B][Hkv][cap][d] view, strided
    q = torch.zeros(B, 8, 128, dtype=torch.float16, device="cuda")
    desc = H.make_desc(q, K)
    k8, ks = _shadow(H, desc, K, [cap, cap])
    H.hill_sync_status()
    codes, scale = oracle_mod.quantize_rows(K.contiguous().cpu())
    assert np.array_equal(k8.cpu().numpy(), codes)
    assert np.array_equal(ks.cpu().numpy()[:, :, :cap], scale)


SHAPES = [
    # B, H, Hkv, cap, lens
    (3, 8, 8, 1000, [1000, 517, 33]),
    (2, 32, 8, 700, [700, 1]),
    (2, 8, 1, 300, [300, 299]),
    (4, 16, 2, 129, [129, 0, 64, 95]),
    (2, 32, 1, 700, [700, 333]),   # 32 query heads on one KV head
    (2, 28, 4, 300, [300, 150]),   # 7 query heads per KV head
    (2, 40, 40, 200, [200, 77]),   # 40 KV heads: two scoring passes
]


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_score_f8_matches_oracle(H, oracle_mod, mode, dtype, shape):
    B, Hq, Hkv, cap, lens = shape
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=dtype, seed=cap + Hq)
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    k8, ks = _shadow(H, desc, K, lens)
    ws = H.alloc_workspace(desc, mode, 0)
    s = torch.zeros(B, cap, device="cuda")
    H.hill_score_f8(desc, q, k8, ks, lens_t, mode, s, ws=ws)
    H.hill_sync_status()
    codes, scale = oracle_mod.quantize_rows(K.cpu())
    z8 = oracle_mod.logits_q8(q.cpu(), codes, scale, lens)
    check_scores(s.cpu().numpy(), oracle_mod.scores(mode, z8, lens), lens)


# Shapes that take the tensor-core E4M3 kernel (2 to 16 query heads per KV
# head and at least 64 MB of codes per call): G = 4 on one 64K-token sequence,
# G = 2 with two ragged sequences, G = 2 with three (one of a single token)
TC_SHAPES = [
    # B, H, Hkv, cap, lens
    (1, 32, 8, 65600, [65537]),
    (2, 32, 16, 33000, [33000, 20001]),
    (3, 16, 8, 22000, [22000, 1, 15031]),
]


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
@pytest.mark.parametrize("shape", TC_SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_score_f8_tensor_core_matches_oracle(H, oracle_mod, mode, dtype, shape):
    """hill_score_f8 and the split step's E4M3 K stream on shapes the
    tensor-core kernel takes, against the oracle's scores on the 8-bit
    operands; the split step's selection exact on its own scores."""
    B, Hq, Hkv, cap, lens = shape
    assert B * cap * Hkv * 128 >= 64 << 20
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=dtype, seed=cap + 5 * Hq,
                                         kind="zipf" if mode == ATTN else "normal")
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    k8, ks = _shadow(H, desc, K, lens)
    codes, scale = oracle_mod.quantize_rows(K.cpu())
    ref = oracle_mod.scores(mode, oracle_mod.logits_q8(q.cpu(), codes, scale, lens), lens)
    ws = H.alloc_workspace(desc, mode, 0)
    s = torch.full((B, cap), float("nan"), device="cuda")
    H.hill_score_f8(desc, q, k8, ks, lens_t, mode, s, ws=ws)
    H.hill_sync_status()
    check_scores(s.cpu().numpy(), ref, lens)
    k = [max(1, n // 10) for n in lens]
    max_k = max(k)
    wss = H.alloc_workspace(desc, mode, max_k)
    s2 = torch.full((B, cap), float("nan"), device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    kt = torch.tensor(k, dtype=torch.int32, device="cuda")
    H.hill_evict_step_begin_f8(desc, q, k8, ks, lens_t, max_k, mode, None, s2, wss)
    H.hill_evict_step_end(desc, lens_t, kt, max_k, mode, None, s2, idx, cnt, wss)
    H.hill_sync_status()
    check_scores(s2.cpu().numpy(), ref, lens, what="split step")
    idx_o, cnt_o, _ = oracle_mod.topk(s2.cpu().numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_score_f8_long(H, oracle_mod, mode):
    """Long sequences: many tiles per scoring CTA, and (ATTN) the
    normalisation with more than two CTAs per SM, which first combines the
    partials once per (sequence, head)."""
    B, Hq, Hkv, cap = 2, 8, 8, 40000
    lens = [40000, 23457]
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=404)
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    k8, ks = _shadow(H, desc, K, lens)
    ws = H.alloc_workspace(desc, mode, 0)
    s = torch.zeros(B, cap, device="cuda")
    H.hill_score_f8(desc, q, k8, ks, lens_t, mode, s, ws=ws)
    H.hill_sync_status()
    codes, scale = oracle_mod.quantize_rows(K.cpu())
    z8 = oracle_mod.logits_q8(q.cpu(), codes, scale, lens)
    check_scores(s.cpu().numpy(), oracle_mod.scores(mode, z8, lens), lens)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_evict_step_f8(H, oracle_mod, mode):
    """Selection from the shadow against the oracle's 8-bit scores (gap rule),
    attention on the original keys and values against the oracle on the GPU's
    own index set, and scoring-only calls without the 16-bit caches."""
    B, Hq, Hkv, cap = 3, 8, 2, 1200
    lens, k = [1200, 777, 50], [240, 155, 10]
    max_k = 240
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=33, kind="zipf")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K, V)
    k8, ks = _shadow(H, desc, K, lens)
    ws = H.alloc_workspace(desc, mode, max_k)
    scores = torch.zeros(B, cap, device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    out = torch.empty(B, Hq, 128, device="cuda")
    H.hill_evict_step_f8(desc, q, k8, ks, K, V, lens_t, _i32(k), max_k, mode, None, scores, idx, cnt, out, ws)
    idx2 = torch.empty_like(idx)
    cnt2 = torch.empty_like(cnt)
    H.hill_evict_step_f8(desc, q, k8, ks, None, None, lens_t, _i32(k), max_k, mode, None, None, idx2, cnt2, None,
                         ws)
    H.hill_sync_status()
    assert torch.equal(idx, idx2) and torch.equal(cnt, cnt2)
    codes, scale = oracle_mod.quantize_rows(K.cpu())
    s_ref = oracle_mod.scores(mode, oracle_mod.logits_q8(q.cpu(), codes, scale, lens), lens)
    check_scores(scores.cpu().numpy(), s_ref, lens)
    check_selection(idx.cpu().numpy(), cnt.cpu().numpy(), s_ref, lens, k, max_k)
    o_ref = oracle_mod.sparse_attn(q.cpu(), K.cpu(), V.cpu(), idx.cpu().numpy(), cnt.cpu().numpy())
    check_attn(out.cpu().numpy(), o_ref)


def test_f8_selection_recall_on_workload2(H, oracle_mod):
    """Recall of the shadow's selection against the exact (16-bit) selection
    on one full-size layer of the 4K benchmark workload.  The paper argues
    the low precision only serves the ranking (Sec. 4.4); this measures how
    much of the exact top-20 % it keeps."""
    w = inputs.config(2)
    K, V = inputs.layer_cache(w, 0, device="cuda")
    t = w.steps - 1
    q = inputs.step_query(w, 0, t, device="cuda")
    lens = w.lens_at(t)
    kb = w.budget_at(t)
    lens_t, k_t = _i32(lens), _i32(kb)
    desc = H.make_desc(q, K, V)
    k8, ks = _shadow(H, desc, K, lens)
    ws = H.alloc_workspace(desc, ATTN, w.max_k)
    sel = []
    for f8 in (False, True):
        idx = torch.empty(w.batch, w.max_k, dtype=torch.int32, device="cuda")
        cnt = torch.empty(w.batch, dtype=torch.int32, device="cuda")
        if f8:
            H.hill_evict_step_f8(desc, q, k8, ks, None, None, lens_t, k_t, w.max_k, ATTN, None, None, idx, cnt,
                                 None, ws)
        else:
            H.hill_evict_step(desc, q, K, V, lens_t, k_t, w.max_k, ATTN, None, None, idx, cnt, None, ws)
        sel.append((idx.cpu().numpy(), cnt.cpu().numpy()))
    H.hill_sync_status()
    hit = tot = 0
    for b in range(w.batch):
        a = set(sel[0][0][b, : sel[0][1][b]].tolist())
        c = set(sel[1][0][b, : sel[1][1][b]].tolist())
        hit += len(a & c)
        tot += len(a)
    recall = hit / tot
    print(f"E4M3 shadow recall of the exact top-k on workload 2: {recall:.4f}")
    assert recall > 0.9

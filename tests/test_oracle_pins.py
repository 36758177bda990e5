"""Pins for the CPU oracle: each check ties the oracle to something other than
itself -- a library routine, a closed form, an invariant of the method, a
brute force on tiny inputs or a hand-derived case -- so that a dropped term, a
wrong sign or index, or a transposed operand in oracle/hill_oracle.c fails at
least one of them.  CPU only.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from paper_2602_18750_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "tiny_cases.json")


def _expr(v):
    return eval(str(v), {"__builtins__": {}}, {"e": math.e, "exp": math.exp})


def _exact(oracle_mod, t):
    return oracle_mod.decode16(t)


def _expand_kv(x, H):
    """[B][Hkv][cap][d] -> [B][H][cap][d] with the contiguous head grouping
    (query head h reads KV head h // (H/Hkv)), via torch.repeat_interleave."""
    return torch.repeat_interleave(x, H // x.shape[1], dim=1)


# ---------------------------------------------------------------- decoding
def test_decode_f16_all_bit_patterns(oracle_mod):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = oracle_mod.decode16(bits, dtype=oracle_mod.F16)
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


def test_decode_bf16_all_bit_patterns(oracle_mod):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = oracle_mod.decode16(bits, dtype=oracle_mod.BF16)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


# ---------------------------------------------------------------- golden
@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_golden_hand_derived(oracle_mod, case, dtype):
    q = torch.tensor(case["q"], dtype=dtype)
    K = torch.tensor(case["K"], dtype=dtype)
    V = torch.tensor(case["V"], dtype=dtype)
    lens, k, max_k = case["lens"], case["k"], case["max_k"]
    z = oracle_mod.logits(q, K, lens)
    for b, n in enumerate(lens):
        for h in range(case["H"]):
            want = [_expr(x) for x in case["z"][b][h]]
            assert np.allclose(z[b, h, :n], want, rtol=0, atol=1e-15)
            assert np.all(np.isnan(z[b, h, n:]))
    for mode, key in ((oracle_mod.ATTN, "attn"), (oracle_mod.RAW, "raw")):
        s = oracle_mod.scores(mode, z, lens)
        for b, n in enumerate(lens):
            want = [_expr(x) for x in case[f"s_{key}"][b]]
            assert np.allclose(s[b, :n], want, rtol=1e-14, atol=1e-15)
        idx, count, rc = oracle_mod.topk(s, lens, k, max_k)
        assert rc == 0
        assert idx.tolist() == case[f"idx_{key}"]
        assert count.tolist() == case["count"]
        r = oracle_mod.evict_step(mode, q, K, V, lens, k, max_k)
        assert r["rc"] == 0 and r["idx"].tolist() == case[f"idx_{key}"]
        if key == "attn":
            want = np.array([[[_expr(x) for x in row] for row in hb] for hb in case["out_attn"]])
            assert np.allclose(r["out"], want, rtol=1e-14, atol=1e-15)


# ---------------------------------------------------------------- logits
@pytest.mark.parametrize("H,Hkv,d", [(8, 8, 128), (8, 2, 64), (4, 1, 128), (6, 3, 32),
                                     (28, 4, 128), (12, 1, 64), (40, 40, 128)])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_logits_match_torch_fp64_matmul(oracle_mod, H, Hkv, d, dtype):
    B, cap = 3, 70
    lens = [70, 33, 0]
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, lens, dtype=dtype, seed=11)
    z = oracle_mod.logits(q, K, lens)
    ref = torch.matmul(_expand_kv(K.double(), H), q.double().unsqueeze(-1)).squeeze(-1) / math.sqrt(d)
    for b, n in enumerate(lens):
        assert np.allclose(z[b, :, :n], ref[b, :, :n].numpy(), rtol=1e-12, atol=1e-12)
        assert np.all(np.isnan(z[b, :, n:]))


# ---------------------------------------------------------------- importance
def test_attn_single_head_is_torch_softmax(oracle_mod):
    B, H, d, cap = 2, 1, 128, 90
    lens = [90, 41]
    q, K, V, _ = inputs.random_case(B, H, H, d, cap, lens, seed=3, kind="zipf")
    z = oracle_mod.logits(q, K, lens)
    s = oracle_mod.scores(oracle_mod.ATTN, z, lens)
    for b, n in enumerate(lens):
        ref = torch.softmax(torch.from_numpy(z[b, 0, :n]), dim=0).numpy()
        assert np.allclose(s[b, :n], ref, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("H,Hkv", [(8, 8), (8, 2), (4, 1)])
def test_attn_is_sum_of_torch_softmax_rows(oracle_mod, H, Hkv):
    B, d, cap = 2, 64, 57
    lens = [57, 19]
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, lens, seed=5, kind="zipf" if H == Hkv else "normal")
    z = oracle_mod.logits(q, K, lens)
    s = oracle_mod.scores(oracle_mod.ATTN, z, lens)
    for b, n in enumerate(lens):
        p = torch.softmax(torch.from_numpy(z[b, :, :n]), dim=-1)
        assert np.allclose(s[b, :n], p.sum(0).numpy(), rtol=1e-12, atol=1e-15)
        # invariants: every weight is a probability and each head contributes mass 1
        assert np.isclose(s[b, :n].sum(), H, rtol=1e-12)
        assert np.all(s[b, :n] >= 0) and np.all(s[b, :n] <= H)
        assert np.all(np.isnan(s[b, n:]))


def test_raw_mqa_closed_form(oracle_mod):
    """MQA (one KV head): sum_h q_h.K_j/sqrt(d) = (sum_h q_h).K_j/sqrt(d)."""
    B, H, d, cap = 2, 6, 128, 40
    lens = [40, 13]
    q, K, V, _ = inputs.random_case(B, H, 1, d, cap, lens, seed=9)
    s = oracle_mod.scores(oracle_mod.RAW, oracle_mod.logits(q, K, lens), lens)
    qx, Kx = _exact(oracle_mod, q), _exact(oracle_mod, K)
    for b, n in enumerate(lens):
        ref = Kx[b, 0, :n] @ qx[b].sum(0) / math.sqrt(d)
        assert np.allclose(s[b, :n], ref, rtol=1e-12, atol=1e-12)


def test_raw_gqa_group_sums(oracle_mod):
    """GQA: RAW importance equals sum over KV heads g of (sum of the G query
    heads of g) . K_g,j / sqrt(d) -- pins the head -> KV-head map."""
    B, H, Hkv, d, cap = 1, 8, 2, 32, 25
    lens = [25]
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, lens, seed=21)
    s = oracle_mod.scores(oracle_mod.RAW, oracle_mod.logits(q, K, lens), lens)
    qx, Kx = _exact(oracle_mod, q), _exact(oracle_mod, K)
    G = H // Hkv
    ref = sum(Kx[0, g] @ qx[0, g * G:(g + 1) * G].sum(0) for g in range(Hkv)) / math.sqrt(d)
    assert np.allclose(s[0], ref, rtol=1e-12, atol=1e-12)
    # a transposed grouping (h -> h % Hkv) gives a different answer on this input
    wrong = sum(Kx[0, g] @ qx[0, g::Hkv].sum(0) for g in range(Hkv)) / math.sqrt(d)
    assert not np.allclose(s[0], wrong, rtol=1e-6)


def test_accumulation_mass_over_steps(oracle_mod):
    """Running importance: after t steps of ATTN, sum_j A[b,j] = H * t."""
    B, H, d, cap, steps = 2, 4, 64, 30, 5
    A = np.zeros((B, cap))
    _, K, V, _ = inputs.random_case(B, H, H, d, cap, [30, 30], seed=2)
    for t in range(steps):
        lens = [20 + t, 10 + 2 * t]
        q = inputs.step_query(inputs.config(2, layers=1, batch=B, heads=H, kv_heads=H, head_dim=d,
                                            prompt_lens=(20, 10), steps=steps), 0, t)
        s = oracle_mod.scores(oracle_mod.ATTN, oracle_mod.logits(q, K, lens), lens)
        A_new = oracle_mod.accumulate(s, A, lens)
        for b, n in enumerate(lens):
            assert np.allclose(A_new[b, :n] - A[b, :n], s[b, :n], rtol=0, atol=1e-15)
            assert np.array_equal(A_new[b, n:], A[b, n:])
        A = A_new
    assert np.allclose(A.sum(1), H * steps, rtol=1e-12)


# ---------------------------------------------------------------- top-k
def _brute_topk(key, n, k):
    order = sorted(range(n), key=lambda j: (-key[j], j))
    return sorted(order[: max(0, min(k, n))])


def test_topk_brute_force_and_torch_values(oracle_mod):
    rng = np.random.default_rng(0)
    B, cap = 6, 64
    key = rng.standard_normal((B, cap))
    key[1, 10:20] = 0.5                      # a block of exact ties
    key[2] = np.round(key[2])                # heavy ties
    lens = [64, 40, 64, 1, 0, 17]
    k = [13, 15, 30, 5, 3, 17]
    max_k = 32
    idx, count, rc = oracle_mod.topk(key, lens, k, max_k)
    assert rc == 0
    for b in range(B):
        want = _brute_topk(key[b], lens[b], k[b])
        assert count[b] == len(want) == min(k[b], lens[b])
        assert idx[b, : count[b]].tolist() == want
        assert np.all(idx[b, count[b]:] == -1)
        if lens[b] and k[b]:
            tv = torch.topk(torch.from_numpy(key[b, : lens[b]]), min(k[b], lens[b])).values
            assert sorted(key[b, want].tolist()) == sorted(tv.tolist())


def test_topk_special_budgets(oracle_mod):
    rng = np.random.default_rng(1)
    key = rng.standard_normal((3, 50))
    lens = [50, 50, 30]
    idx, count, rc = oracle_mod.topk(key, lens, [50, 0, 99], 50)
    assert rc == 0
    assert idx[0].tolist() == list(range(50))           # k = len: everything
    assert count[1] == 0 and np.all(idx[1] == -1)       # k = 0: nothing
    assert idx[2, :30].tolist() == list(range(30))      # k > len clamps to len
    idx, count, rc = oracle_mod.topk(key, lens, [40, 40, 40], 8)
    assert rc == 2 and count.tolist() == [8, 8, 8]      # capped by max_k, reported


def test_topk_ties_go_to_lower_index(oracle_mod):
    key = np.zeros((1, 12))
    key[0, [3, 7, 9]] = 2.0
    idx, count, _ = oracle_mod.topk(key, [12], [5], 5)
    assert idx[0].tolist() == [0, 1, 3, 7, 9]
    key[0, 5] = -0.0                         # signed zero ties with +0
    idx, count, _ = oracle_mod.topk(key, [12], [5], 5)
    assert idx[0].tolist() == [0, 1, 3, 7, 9]


def test_topk_nan_ranks_last(oracle_mod):
    key = np.array([[np.nan, 1.0, -5.0, np.nan, 0.0]])
    idx, count, _ = oracle_mod.topk(key, [5], [3], 5)
    assert idx[0, :3].tolist() == [1, 2, 4]


# ---------------------------------------------------------------- E4M3 shadow (Sec. 4.4)
def test_e4m3_decode_all_codes_matches_torch(oracle_mod):
    codes = np.arange(256, dtype=np.uint8)
    got = oracle_mod.e4m3_decode(codes)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan) and nan.sum() == 2
    assert np.array_equal(got[~nan], ref[~nan])
    assert got[0x7E] == 448.0 and got[0x01] == 2.0 ** -9 and got[0x08] == 2.0 ** -6


def test_e4m3_encode_round_trip_ties_and_torch(oracle_mod):
    codes = np.array([c for c in range(256) if (c & 0x7F) != 0x7F], dtype=np.uint8)
    vals = oracle_mod.e4m3_decode(codes)
    assert np.array_equal(oracle_mod.e4m3_encode(vals.astype(np.float32)), codes)     # round trip
    pos = np.sort(np.unique(vals[vals > 0]))
    mids = (pos[:-1] + pos[1:]) / 2                    # exact midpoints (float32-representable)
    enc = oracle_mod.e4m3_encode(mids.astype(np.float32))
    lo = oracle_mod.e4m3_encode(pos[:-1].astype(np.float32))
    hi = oracle_mod.e4m3_encode(pos[1:].astype(np.float32))
    assert np.all(enc == np.where(lo % 2 == 0, lo, hi))                            # ties to the even code
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.uniform(-463, 463, 20000), rng.uniform(-0.02, 0.02, 20000),
                        [448.0, -0.0]]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(oracle_mod.e4m3_encode(x), ref)
    # beyond the last rounding interval torch's cast gives NaN; the encoder
    # (like the kernel's saturating conversion) gives +-448
    assert oracle_mod.e4m3_encode(np.array([500.0, -1e4, 3e38], np.float32)).tolist() == [0x7E, 0xFE, 0x7E]


def test_quantize_rows_bounds(oracle_mod):
    g = torch.Generator().manual_seed(4)
    x = (torch.randn(64, 128, generator=g) * torch.logspace(-3, 2, 64)[:, None]).half()
    x[5] = 0.0
    codes, scale = oracle_mod.quantize_rows(x)
    xd = oracle_mod.decode16(x)
    amax = np.abs(xd).max(axis=1)
    assert scale[5] == 0.0 and np.all(codes[5] == 0)
    for r in range(64):
        if r == 5:
            continue
        assert scale[r] == np.float32(np.float32(amax[r]) / np.float32(448.0))
        dec = oracle_mod.e4m3_decode(codes[r])
        y = xd[r] * np.float64(np.float32(448.0) / np.float32(amax[r]))
        assert np.abs(dec).max() == 448.0
        # E4M3 rounding error: half a spacing, i.e. 1/16 relative above 2^-6, 2^-10 below
        assert np.all(np.abs(dec - y) <= np.maximum(np.abs(y) / 16, 2.0 ** -10) * (1 + 1e-6))


@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_quantize_rows_matches_torch_float32_steps_and_e4m3_cast(oracle_mod, dtype):
    """Sec. 4.4's key shadow, row by row, computed here with torch alone: the
    row maximum |x| in float32, its reciprocal 448 / amax and the products
    x * (448 / amax) as float32 tensor operations, saturated to +-448, then
    torch's own cast to float8_e4m3fn; the scale is amax / 448 in float32.
    The oracle's codes and scales must equal these bit for bit, so a step the
    oracle and the kernel might share by mistake (a scale of 448 / amax the
    other way round, rounding the product in double, truncating instead of
    rounding, a lost sign) fails here."""
    g = torch.Generator().manual_seed(41)
    n, d = 600, 128
    mag = torch.logspace(-5, 4, n)                                 # row magnitudes across the dtypes' range
    x = (torch.randn(n, d, generator=g) * mag[:, None]).to(dtype)
    x[7] = 0.0                                                     # an all-zero row
    x[8] = 0.0
    x[8, 3] = -2.5                                                 # one negative entry holds the maximum
    x[9, :] = x[9, :].abs().neg()                                  # every entry negative
    x[10, ::2] = 0.0
    codes, scale = oracle_mod.quantize_rows(x)
    xf = x.float()
    amax = xf.abs().amax(dim=1)
    nz = amax > 0
    r = torch.full_like(amax, 448.0)
    r[nz] = torch.tensor(448.0, dtype=torch.float32) / amax[nz]
    y = (xf * r[:, None]).clamp(-448.0, 448.0)
    ref_codes = y.to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    ref_codes[~nz.numpy()] = 0
    ref_scale = torch.where(nz, amax / torch.tensor(448.0, dtype=torch.float32), torch.zeros_like(amax)).numpy()
    assert np.array_equal(codes, ref_codes), f"{(codes != ref_codes).sum()} codes differ"
    assert np.array_equal(scale.view(np.uint32), ref_scale.view(np.uint32))
    assert codes[8, 3] == 0xFE and np.all(codes[9][codes[9] != 0x80] >= 0x80)


def test_logits_q8_is_fp64_matmul_of_dequantized(oracle_mod):
    B, H, Hkv, d, cap = 2, 8, 2, 128, 40
    lens = [40, 23]
    q, K, _, _ = inputs.random_case(B, H, Hkv, d, cap, lens, seed=8)
    kc, ks = oracle_mod.quantize_rows(K)
    qc, qs = oracle_mod.quantize_rows(q)
    Kd = torch.from_numpy(oracle_mod.e4m3_decode(kc) * ks[..., None].astype(np.float64))
    qd = torch.from_numpy(oracle_mod.e4m3_decode(qc) * qs[..., None].astype(np.float64))
    ref = torch.matmul(_expand_kv(Kd, H), qd.unsqueeze(-1)).squeeze(-1) / math.sqrt(d)
    z8 = oracle_mod.logits_q8(q, kc, ks, lens)
    for b in range(B):
        assert np.allclose(z8[b, :, : lens[b]], ref[b, :, : lens[b]].numpy(), rtol=1e-12, atol=1e-12)
        assert np.all(np.isnan(z8[b, :, lens[b]:]))


def test_logits_q8_lossless_rows_equal_exact_logits(oracle_mod):
    """Rows built from E4M3 values times 2^-4 whose largest magnitude is 448 * 2^-4
    quantise without loss, so the 8-bit logits equal the exact ones."""
    rng = np.random.default_rng(9)
    grid = oracle_mod.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))
    grid = grid[grid >= 2.0 ** -6]                     # normals: exact in binary16 after the 2^-4 shift
    B, H, Hkv, d, cap = 1, 4, 2, 128, 17

    def rows(n):
        v = rng.choice(grid, size=(n, d)) * rng.choice([-1.0, 1.0], size=(n, d))
        v[np.arange(n), rng.integers(0, d, n)] = 448.0
        return torch.from_numpy(v * 2.0 ** -4).half()

    q = rows(B * H).reshape(B, H, d)
    K = rows(B * Hkv * cap).reshape(B, Hkv, cap, d)
    kc, ks = oracle_mod.quantize_rows(K)
    assert np.all(ks == np.float32(28.0 / 448.0))
    z8 = oracle_mod.logits_q8(q, kc, ks, [cap])
    z = oracle_mod.logits(q, K, [cap])
    assert np.allclose(z8, z, rtol=1e-12, atol=0)


# ---------------------------------------------------------------- per-KV-head selection
def test_kvh_reduces_to_sequence_path_for_one_kv_head(oracle_mod):
    """With Hkv = 1 the per-KV-head scores, selection and attention are the
    per-sequence ones."""
    B, H, d, cap = 2, 4, 64, 50
    lens, k = [50, 31], [9, 31]
    q, K, V, _ = inputs.random_case(B, H, 1, d, cap, lens, seed=14)
    z = oracle_mod.logits(q, K, lens)
    for mode in (oracle_mod.ATTN, oracle_mod.RAW):
        s1 = oracle_mod.scores_kvh(mode, z, lens, 1)
        s0 = oracle_mod.scores(mode, z, lens)
        assert np.allclose(s1[:, 0], s0, equal_nan=True, rtol=0, atol=0)
        i1, c1, _ = oracle_mod.topk_kvh(s1, lens, k, 32)
        i0, c0, _ = oracle_mod.topk(s0, lens, k, 32)
        assert np.array_equal(i1[:, 0], i0) and np.array_equal(c1[:, 0], c0)
        o1 = oracle_mod.sparse_attn_kvh(q, K, V, i1, c1)
        o0 = oracle_mod.sparse_attn(q, K, V, i0, c0)
        assert np.array_equal(o1, o0)


def test_kvh_mha_selects_each_heads_own_softmax_top(oracle_mod):
    """MHA (G = 1), ATTN: each KV head keeps the top-k of its own softmax row,
    which is the top-k of its logits (softmax is monotone) -- checked against
    torch.topk on the logits; the per-head mass is 1 (Σ_j p = 1)."""
    B, H, d, cap = 1, 6, 64, 40
    lens, k = [40], [7]
    q, K, V, _ = inputs.random_case(B, H, H, d, cap, lens, seed=15)
    z = oracle_mod.logits(q, K, lens)
    s = oracle_mod.scores_kvh(oracle_mod.ATTN, z, lens, H)
    assert np.allclose(s[0].sum(axis=1), 1.0)
    idx, cnt, _ = oracle_mod.topk_kvh(s, lens, k, 7)
    for g in range(H):
        want = sorted(torch.topk(torch.from_numpy(z[0, g]), 7).indices.tolist())
        assert idx[0, g].tolist() == want


@pytest.mark.parametrize("H,Hkv", [(14, 2), (12, 1)])
def test_kvh_attn_group_sums_of_torch_softmax(oracle_mod, H, Hkv):
    """Groups that are not a power of two (7) or above 8 heads (12): the
    per-KV-head ATTN importance is the sum of the torch softmax rows of
    exactly the G query heads h // G = g, each group carrying mass G."""
    B, d, cap = 2, 64, 45
    lens = [45, 17]
    G = H // Hkv
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, lens, seed=23)
    z = oracle_mod.logits(q, K, lens)
    s = oracle_mod.scores_kvh(oracle_mod.ATTN, z, lens, Hkv)
    for b, n in enumerate(lens):
        p = torch.softmax(torch.from_numpy(z[b, :, :n]), dim=-1).numpy()
        for g in range(Hkv):
            assert np.allclose(s[b, g, :n], p[g * G:(g + 1) * G].sum(0), rtol=1e-12, atol=1e-15)
            assert np.isclose(s[b, g, :n].sum(), G, rtol=1e-12)


def test_kvh_attention_uses_each_heads_rows(oracle_mod):
    """GQA: query heads of KV head g attend over idx[b][g] only -- a one-token
    set gives that token's V row of head g for all G query heads."""
    B, H, Hkv, d, cap = 1, 4, 2, 32, 12
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, [12], seed=16)
    idx = np.array([[[3, 0], [10, 0]]], dtype=np.int32)
    cnt = np.array([[1, 1]], dtype=np.int32)
    o = oracle_mod.sparse_attn_kvh(q, K, V, idx, cnt)
    Vd = oracle_mod.decode16(V)
    for h in range(H):
        g = h // 2
        assert np.allclose(o[0, h], Vd[0, g, idx[0, g, 0]])


# ---------------------------------------------------------------- BKP bookkeeping (Sec. 4.2)
def test_bkp_without_window_is_topk(oracle_mod):
    """recent = 0 reduces BKP selection to the pinned top-k, and the hit table
    gains exactly one count at every kept token."""
    rng = np.random.default_rng(11)
    key = np.round(rng.standard_normal((5, 40)), 1)
    lens, k = [40, 33, 1, 0, 25], [7, 33, 4, 2, 0]
    hits0 = rng.integers(0, 50, size=(5, 40)).astype(np.uint16)
    idx, count, rc, hits = oracle_mod.bkp_select(key, lens, k, 0, 40, hits0)
    idx2, count2, rc2 = oracle_mod.topk(key, lens, k, 40)
    assert rc == rc2 == 0 and np.array_equal(idx, idx2) and np.array_equal(count, count2)
    want = hits0.astype(np.int64)
    for b in range(5):
        want[b, idx[b, : count[b]]] += 1
    assert np.array_equal(hits.astype(np.int64), want)


def test_bkp_window_and_exchange_property(oracle_mod):
    """The kept set is the pinned window [len-R, len) plus a ranked set T of
    min(k, len-R) older tokens such that no older token outside T beats one
    inside it in (key desc, index asc) -- checked pair by pair, which fixes T
    uniquely without sorting."""
    rng = np.random.default_rng(12)
    for trial in range(60):
        cap = int(rng.integers(1, 14))
        key = np.round(rng.standard_normal((1, cap)) * 2) / 2        # many ties
        ln = int(rng.integers(0, cap + 1))
        R_req = int(rng.integers(0, cap + 3))
        kb = int(rng.integers(0, cap + 3))
        idx, count, rc, _ = oracle_mod.bkp_select(key, [ln], [kb], R_req, cap + 4)
        assert rc == 0
        R = min(R_req, ln)
        older = ln - R
        got = idx[0, : count[0]].tolist()
        assert got == sorted(got) and np.all(idx[0, count[0]:] == -1)
        assert count[0] == R + min(kb, older)
        assert got[len(got) - R:] == list(range(older, ln))          # the window, last
        T = set(got[: len(got) - R])
        assert all(j < older for j in T)
        for i in T:
            for j in range(older):
                if j not in T:
                    assert key[0, i] > key[0, j] or (key[0, i] == key[0, j] and i < j)


def test_bkp_hits_count_steps_and_saturate(oracle_mod):
    """Over several decode steps the table counts, per token, the steps that
    kept it (tallied from the returned index sets), and stops at 65535."""
    rng = np.random.default_rng(13)
    cap, steps = 30, 9
    hits = np.zeros((2, cap), dtype=np.uint16)
    tally = np.zeros((2, cap), dtype=np.int64)
    for t in range(steps):
        key = rng.standard_normal((2, cap))
        lens = [20 + t, 12 + t]
        idx, count, rc, hits = oracle_mod.bkp_select(key, lens, [5, 3], 4, 16, hits)
        assert rc == 0
        for b in range(2):
            tally[b, idx[b, : count[b]]] += 1
    assert np.array_equal(hits.astype(np.int64), tally)
    full = np.full((1, 6), 65534, dtype=np.uint16)
    for _ in range(3):
        _, _, _, full = oracle_mod.bkp_select(np.zeros((1, 6)), [6], [6], 0, 6, full)
    assert np.all(full == 65535)


def test_bkp_budget_cap_keeps_most_recent(oracle_mod):
    """A window wider than max_k keeps its most recent tokens; otherwise the
    ranked part gets what the window leaves; both report rc 2."""
    key = np.arange(10, dtype=np.float64)[None, :]
    idx, count, rc, _ = oracle_mod.bkp_select(key, [10], [3], 6, 4)
    assert rc == 2 and count[0] == 4 and idx[0].tolist() == [6, 7, 8, 9]
    # window [8, 9] first, then the best 2 of the older tokens: 6 and 7
    idx, count, rc, _ = oracle_mod.bkp_select(key, [10], [3], 2, 4)
    assert rc == 2 and idx[0].tolist() == [6, 7, 8, 9]


def test_cec_single_head_raw_equals_attn_selection(oracle_mod):
    """Sec. 4.4: for one head and one step, ranking by raw q.K equals ranking by
    softmax weight (softmax is monotonic), so both modes select the same set."""
    for seed in range(4):
        q, K, V, _ = inputs.random_case(2, 1, 1, 128, 300, [300, 257], seed=seed, kind="zipf")
        lens, k = [300, 257], [60, 25]
        ra = oracle_mod.evict_step(oracle_mod.ATTN, q, K, V, lens, k, 64, with_attn=False)
        rr = oracle_mod.evict_step(oracle_mod.RAW, q, K, V, lens, k, 64, with_attn=False)
        assert np.array_equal(ra["idx"], rr["idx"])


@pytest.mark.parametrize("mode", [0, 1])
def test_planted_heavy_hitters_always_selected(oracle_mod, mode):
    """The heavy-hitter workload (64 planted keys, 4x along q) at reduced size:
    every planted token is in the selected set in both modes."""
    w = inputs.config(1, heads=4, kv_heads=4, prompt_lens=(512,), planted=16, budget_tokens=64)
    K, V = inputs.layer_cache(w, 0)
    q = inputs.step_query(w, 0, 0)
    # recover the planted positions from the generator's construction: their
    # projection on the query direction is 4*sqrt(d) for every head
    qx = oracle_mod.decode16(q)[0]
    Kx = oracle_mod.decode16(K)[0]
    proj = np.stack([Kx[h] @ (qx[h] / np.linalg.norm(qx[h])) for h in range(4)])
    planted = np.where((proj > 2.0 * math.sqrt(128)).all(0))[0]
    assert len(planted) == 16
    r = oracle_mod.evict_step(mode, q, K, V, [512], [64], 64, with_attn=False)
    assert set(planted.tolist()) <= set(r["idx"][0, : r["count"][0]].tolist())


# ---------------------------------------------------------------- attention
@pytest.mark.parametrize("H,Hkv", [(8, 8), (8, 2), (4, 1)])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_full_budget_equals_dense_sdpa(oracle_mod, H, Hkv, dtype):
    """k = len selects every token, so the sparse attention is the dense decode
    attention: torch scaled_dot_product_attention in float64."""
    B, d, cap = 2, 64, 45
    lens = [45, 22]
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, lens, dtype=dtype, seed=4)
    r = oracle_mod.evict_step(oracle_mod.ATTN, q, K, V, lens, lens, cap)
    Ke, Ve = _expand_kv(K.double(), H), _expand_kv(V.double(), H)
    for b, n in enumerate(lens):
        ref = torch.nn.functional.scaled_dot_product_attention(
            q[b].double().unsqueeze(1), Ke[b, :, :n], Ve[b, :, :n]).squeeze(1)
        assert np.allclose(r["out"][b], ref.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_special_cases(oracle_mod):
    B, H, Hkv, d, cap = 2, 4, 2, 32, 20
    q, K, V, _ = inputs.random_case(B, H, Hkv, d, cap, [20, 20], seed=8)
    Vx = oracle_mod.decode16(V)
    # one selected token: the output is exactly that token's value row
    idx = np.array([[7], [13]], dtype=np.int32)
    out = oracle_mod.sparse_attn(q, K, V, idx, [1, 1])
    for b in range(B):
        for h in range(H):
            assert np.array_equal(out[b, h], Vx[b, h // 2, idx[b, 0]])
    # a constant value cache gives that constant whatever the weights
    Vc = torch.full_like(V, 1.5)
    idx = np.array([[0, 3, 9, 19], [2, 4, 6, 8]], dtype=np.int32)
    out = oracle_mod.sparse_attn(q, K, Vc, idx, [4, 3])
    assert np.allclose(out, 1.5, rtol=0, atol=1e-15)
    # empty selection gives zero
    out = oracle_mod.sparse_attn(q, K, V, idx, [0, 0])
    assert np.all(out == 0)
    # the order of the index list does not matter
    a = oracle_mod.sparse_attn(q, K, V, idx, [4, 4])
    b = oracle_mod.sparse_attn(q, K, V, idx[:, ::-1].copy(), [4, 4])
    assert np.allclose(a, b, rtol=1e-14, atol=1e-15)


def test_attention_rejects_out_of_range_index(oracle_mod):
    q, K, V, _ = inputs.random_case(1, 2, 2, 16, 10, [10], seed=1)
    with pytest.raises(ValueError):
        oracle_mod.sparse_attn(q, K, V, np.array([[3, 10]], dtype=np.int32), [2])


# ---------------------------------------------------------------- planted mistakes
def test_pins_catch_planted_mistakes(oracle_mod):
    """Plant plausible mistakes on the CPU side (wrong scale, transposed
    operand, softmax over the wrong range) and check that the same pins used
    above reject them."""
    B, H, d, cap = 1, 4, 64, 30
    lens = [21]
    q, K, V, _ = inputs.random_case(B, H, H, d, cap, lens, seed=6)
    z = oracle_mod.logits(q, K, lens)
    ref = torch.matmul(K.double(), q.double().unsqueeze(-1)).squeeze(-1) / math.sqrt(d)
    assert np.allclose(z[0, :, :21], ref[0, :, :21].numpy())
    # missing 1/sqrt(d)
    assert not np.allclose(z[0, :, :21] * math.sqrt(d), ref[0, :, :21].numpy())
    # K read with query and key roles swapped across heads
    zt = oracle_mod.logits(q.flip(1), K, lens)
    assert not np.allclose(zt[0, :, :21], ref[0, :, :21].numpy())
    # softmax over the full capacity instead of the causal row breaks the mass invariant
    zc = np.where(np.isnan(z), 0.0, z)
    s_bad = oracle_mod.scores(oracle_mod.ATTN, zc, [cap])
    assert not np.isclose(s_bad[0, :21].sum(), H)

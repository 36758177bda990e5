"""GPU parity: every CUDA entry point, called through the C ABI, against the
CPU oracle on the same seeded inputs.  Needs a GB300 and the built library.

Sizes run from a handful of tokens to the full benchmark shapes; small cases
span several 32-token tiles with a ragged tail, and the full-size cases use
the same launch path (hill_evict_step) as bench.py on sampled (layer, step)
pairs.
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


def _dev(*ts):
    return [t.cuda() for t in ts]


def _run_step(H, q, K, V, lens, k, max_k, mode, accum=None, with_attn=True):
    ev = H.Evictor(q, K, V, max_k, mode=mode, with_attn=with_attn)
    k_t = torch.tensor(k, dtype=torch.int32, device=q.device)
    ev.step(q, K, V, lens, k_t, accum=accum)
    H.hill_sync_status()
    return ev


def _case(B, Hq, Hkv, cap, lens, dtype, seed, kind="normal", **kw):
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=dtype, seed=seed, kind=kind, **kw)
    return _dev(q, K, V, lens_t)


SHAPES = [
    # B, H, Hkv, cap, lens, k
    (3, 8, 8, 1000, [1000, 517, 33], [200, 103, 40]),
    (2, 32, 8, 700, [700, 1], [64, 5]),
    (2, 8, 1, 300, [300, 299], [30, 299]),
    (4, 4, 2, 129, [129, 0, 64, 95], [13, 3, 64, 0]),
    # fewer query heads than one warp of the normalisation combines
    (2, 2, 1, 300, [300, 150], [30, 15]),
    (2, 1, 1, 257, [257, 100], [20, 100]),
    # groups of more than 8 query heads per KV head (MQA-like): the scoring
    # kernel scores up to 32 from each key tile, the attention up to 16 from
    # each gathered batch (32 = two passes of 16)
    (2, 32, 1, 700, [700, 333], [70, 33]),
    (2, 32, 2, 500, [500, 260], [50, 26]),
    # group sizes that are not powers of two (the kernels' power-of-two group
    # templates with the extra query rows zero), and one of 12 heads (the
    # attention's 16-head template with 4 rows zero)
    (2, 12, 4, 300, [300, 171], [30, 17]),
    (2, 28, 4, 400, [400, 95], [40, 9]),
    (1, 24, 2, 257, [257], [25]),
    # more KV heads than one scoring launch holds (40, as LLaMA-13B): two
    # passes of 20 KV heads
    (2, 40, 40, 300, [300, 130], [60, 26]),
    # few KV heads with large groups deal the tiles to several warps per
    # head: 3 KV heads of 5 query heads take 2 warps each (2 warps idle)
    (3, 15, 3, 300, [300, 5, 240], [30, 5, 24]),
    # one KV head over many short sequences: most warps of a CTA visit no
    # tile of a sequence and leave neutral partials
    (16, 8, 1, 100, [100, 0, 1, 31, 32, 33, 64, 65, 96, 97, 99, 2, 63, 40, 7, 100],
     [10, 0, 1, 3, 3, 3, 6, 6, 9, 9, 9, 1, 6, 4, 1, 10]),
]


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_evict_step_matches_oracle(H, oracle_mod, mode, dtype, shape):
    B, Hq, Hkv, cap, lens, k = shape
    kind = "zipf" if Hq == Hkv else "normal"
    q, K, V, lens_t = _case(B, Hq, Hkv, cap, lens, dtype, seed=100 + cap, kind=kind)
    max_k = max(max(k), 1)
    ev = _run_step(H, q, K, V, lens_t, k, max_k, mode)
    ref = oracle_mod.evict_step(mode, q, K, V, lens, k, max_k, with_attn=False)
    check_scores(ev.scores.cpu().numpy(), ref["s"], lens)
    check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), ref["s"], lens, k, max_k)
    # the selection kernel alone is exact on its own input keys
    idx_o, cnt_o, _ = oracle_mod.topk(ev.scores.cpu().numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(ev.idx.cpu().numpy()[:, :max_k], idx_o)
    assert np.array_equal(ev.count.cpu().numpy(), cnt_o)
    out_ref = oracle_mod.sparse_attn(q, K, V, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
    check_attn(ev.out.cpu().numpy(), out_ref)


@pytest.mark.parametrize("Hkv", [8, 1])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_long_sequences_statistics_kernel(H, oracle_mod, dtype, Hkv):
    """Sequences long enough that the normalisation takes more than two CTAs
    per SM (2 x 157 CTAs on 152 SMs), so the per-head statistics come from
    hill_attn_stats_kernel; accumulation over two steps included.  With one
    KV head the scoring warps deal the tiles (8 partial slots per CTA)."""
    B, Hq, cap = 2, 8, 40000
    lens, k = [40000, 23457], [4000, 2345]
    max_k = 4000
    accum = torch.zeros(B, cap, device="cuda")
    acc_ref = np.zeros((B, cap))
    for step in range(2):
        q, K, V, lens_t = _case(B, Hq, Hkv, cap, lens, dtype, seed=900 + step, kind="zipf")
        ev = _run_step(H, q, K, V, lens_t, k, max_k, ATTN, accum=accum)
        ref = oracle_mod.evict_step(ATTN, q, K, V, lens, k, max_k, with_attn=False)
        check_scores(ev.scores.cpu().numpy(), ref["s"], lens)
        for b in range(B):
            acc_ref[b, : lens[b]] += ref["s"][b, : lens[b]]
    check_scores(accum.cpu().numpy(), acc_ref, lens, what="accum")
    check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), acc_ref, lens, k, max_k)
    out_ref = oracle_mod.sparse_attn(q, K, V, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
    check_attn(ev.out.cpu().numpy(), out_ref)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_separate_calls_equal_fused_step(H, mode):
    q, K, V, lens_t = _case(2, 8, 2, 400, [400, 250], torch.float16, seed=7)
    k = torch.tensor([50, 80], dtype=torch.int32, device="cuda")
    desc = H.make_desc(q, K, V)
    ws = H.alloc_workspace(desc, mode, 80)
    s = torch.zeros(2, 400, device="cuda")
    H.hill_score(desc, q, K, lens_t, mode, s, ws=ws)
    idx = torch.empty(2, 80, dtype=torch.int32, device="cuda")
    cnt = torch.empty(2, dtype=torch.int32, device="cuda")
    H.hill_topk_select(desc, s, lens_t, k, 80, idx, cnt, ws=ws)
    out = torch.empty(2, 8, 128, device="cuda")
    H.hill_gather_sparse_attn(desc, q, K, V, idx, cnt, 80, out, ws=ws)
    ev = H.Evictor(q, K, V, 80, mode=mode)
    ev.step(q, K, V, lens_t, k)
    H.hill_sync_status()
    assert torch.equal(ev.scores[0, :400], s[0, :400]) and torch.equal(ev.scores[1, :250], s[1, :250])
    assert torch.equal(ev.idx, idx) and torch.equal(ev.count, cnt)
    assert torch.equal(ev.out, out)


def test_strided_layouts(H, oracle_mod):
    """Token-major cache [B][cap][Hkv][d] (rows of one head are strided) and a
    query that is a slice of a wider tensor: the per-row copy path."""
    B, Hq, Hkv, cap = 2, 8, 4, 200
    lens, k = [200, 77], [40, 20]
    q0, K0, V0, lens_t = _case(B, Hq, Hkv, cap, lens, torch.float16, seed=31)
    Kt = K0.permute(0, 2, 1, 3).contiguous().permute(0, 2, 1, 3)
    Vt = V0.permute(0, 2, 1, 3).contiguous().permute(0, 2, 1, 3)
    qw = torch.zeros(B, Hq, 256, dtype=q0.dtype, device="cuda")
    qw[:, :, :128] = q0
    qv = qw[:, :, :128]
    assert Kt.stride(2) == Hkv * 128 and qv.stride(1) == 256
    for mode in (ATTN, RAW):
        ev = _run_step(H, qv, Kt, Vt, lens_t, k, 40, mode)
        ref = oracle_mod.evict_step(mode, q0, K0, V0, lens, k, 40, with_attn=False)
        check_scores(ev.scores.cpu().numpy(), ref["s"], lens)
        check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), ref["s"], lens, k, 40)
        out_ref = oracle_mod.sparse_attn(q0, K0, V0, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
        check_attn(ev.out.cpu().numpy(), out_ref)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_accumulation_over_steps(H, oracle_mod, mode):
    """Running importance across decode steps: accum after each step and the
    selection made on it (cumulative importance, Sec. 4.2)."""
    w = inputs.config(5, layers=1, batch=3, prompt_lens=(300, 180, 64), steps=4)
    K, V = inputs.layer_cache(w, 0)
    Kd, Vd = K.cuda(), V.cuda()
    A_gpu = torch.zeros(w.batch, w.capacity, device="cuda")
    A_ref = np.zeros((w.batch, w.capacity))
    max_k = w.max_k
    for t in range(w.steps):
        lens, k = w.lens_at(t), w.budget_at(t)
        q = inputs.step_query(w, 0, t)
        ev = _run_step(H, q.cuda(), Kd, Vd, torch.tensor(lens, dtype=torch.int32, device="cuda"), k,
                       max_k, mode, accum=A_gpu)
        r = oracle_mod.evict_step(mode, q, K, V, lens, k, max_k, accum=A_ref, with_attn=False)
        A_ref = r["accum"]
        check_scores(A_gpu.cpu().numpy(), A_ref, lens, what=f"accum step {t}")
        check_scores(ev.scores.cpu().numpy(), r["s"], lens, what=f"scores step {t}")
        check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), A_ref, lens, k, max_k)


def test_edge_cases(H, oracle_mod):
    # empty sequences, k = 0, k > len, a single token, max_k smaller than k
    q, K, V, lens_t = _case(4, 4, 4, 64, [0, 1, 64, 33], torch.float16, seed=5)
    for mode in (ATTN, RAW):
        ev = _run_step(H, q, K, V, lens_t, [5, 5, 0, 99], 40, mode)
        assert ev.count.cpu().tolist() == [0, 1, 0, 33]
        assert ev.idx[0].eq(-1).all() and ev.idx[2].eq(-1).all()
        assert ev.idx[1, 0].item() == 0 and ev.idx[1, 1:].eq(-1).all()
        assert ev.idx[3, :33].cpu().tolist() == list(range(33))
        out_ref = oracle_mod.sparse_attn(q, K, V, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
        check_attn(ev.out.cpu().numpy(), out_ref)
        assert ev.out[0].eq(0).all() and ev.out[2].eq(0).all()
    # max_k below the budget: count capped at max_k and reported on the device word
    ev = H.Evictor(q, K, V, 8, mode=ATTN)
    ev.step(q, K, V, lens_t, torch.tensor([5, 5, 20, 20], dtype=torch.int32, device="cuda"))
    with pytest.raises(H.HillError) as ei:
        H.hill_sync_status()
    assert ei.value.status == H.HILL_ERR_DEVICE
    assert ev.count.cpu().tolist() == [0, 1, 8, 8]
    H.hill_sync_status()   # the word was cleared


def test_topk_ties_and_signed_zero(H, oracle_mod):
    """Scores with heavy exact ties and -0.0 / +0.0 keys: the selection kernel
    must match the oracle's (score desc, index asc) order exactly."""
    B, cap = 3, 5000
    g = torch.Generator().manual_seed(3)
    s = torch.randint(-3, 4, (B, cap), generator=g).float()
    s[1] = 0.0
    s[1, ::3] = -0.0
    s[2] = torch.randn(cap, generator=g)
    lens, k = [5000, 4999, 1234], [1700, 2500, 617]
    q, K, V, lens_t = _case(B, 4, 4, cap, lens, torch.float16, seed=1)
    desc = H.make_desc(q, K, V)
    idx = torch.empty(B, 2500, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_topk_select(desc, s.cuda(), lens_t, torch.tensor(k, dtype=torch.int32, device="cuda"), 2500, idx, cnt)
    H.hill_sync_status()
    idx_o, cnt_o, _ = oracle_mod.topk(s.numpy().astype(np.float64), lens, k, 2500)
    assert np.array_equal(idx.cpu().numpy(), idx_o)
    assert np.array_equal(cnt.cpu().numpy(), cnt_o)


@pytest.mark.parametrize("cap", [4096 * 3 + 5, 40000, 131072 + 7])
def test_topk_multi_cta_clusters(H, oracle_mod, cap):
    """Capacities that split one sequence over 4 and 8 cluster CTAs."""
    B = 2
    g = torch.Generator().manual_seed(cap)
    s = torch.rand(B, cap, generator=g) ** 4
    lens, k = [cap, cap // 2 + 3], [cap // 10, 2048]
    q, K, V, lens_t = _case(B, 4, 4, 64, [64, 64], torch.float16, seed=1)
    desc = H.make_desc(q, K, V)
    desc.capacity = cap
    max_k = max(k)
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_topk_select(desc, s.cuda(), torch.tensor(lens, dtype=torch.int32, device="cuda"),
                       torch.tensor(k, dtype=torch.int32, device="cuda"), max_k, idx, cnt)
    H.hill_sync_status()
    idx_o, cnt_o, _ = oracle_mod.topk(s.numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(idx.cpu().numpy(), idx_o)
    assert np.array_equal(cnt.cpu().numpy(), cnt_o)


@pytest.mark.parametrize("cap", [40000, 131072 + 7])
def test_topk_cluster_gathered_crossing_bucket(H, oracle_mod, cap):
    """Log-normal scores spread over many octaves, so the bucket of the
    leading 11 key bits that holds the k-th key is small and the cluster
    finishes the search on a gathered copy of it; exact ties planted at the
    k-th score exercise the lowest-index rule there."""
    B = 3
    g = torch.Generator().manual_seed(cap + 1)
    s = torch.exp(torch.randn(B, cap, generator=g) * 4)
    lens, k = [cap, cap - 977, cap // 3], [cap // 5, 3001, 517]
    for b in range(B):
        tau = torch.sort(s[b, : lens[b]], descending=True).values[k[b] - 1]
        pos = torch.randint(0, lens[b], (9,), generator=g)
        s[b, pos] = tau
    q, K, V, lens_t = _case(B, 4, 4, 64, [64, 64, 64], torch.float16, seed=1)
    desc = H.make_desc(q, K, V)
    desc.capacity = cap
    max_k = max(k)
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_topk_select(desc, s.cuda(), torch.tensor(lens, dtype=torch.int32, device="cuda"),
                       torch.tensor(k, dtype=torch.int32, device="cuda"), max_k, idx, cnt)
    H.hill_sync_status()
    idx_o, cnt_o, _ = oracle_mod.topk(s.numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(idx.cpu().numpy(), idx_o)
    assert np.array_equal(cnt.cpu().numpy(), cnt_o)


def test_attention_full_budget_is_dense(H):
    """k = len: the sparse attention is the dense decode attention (checked
    against torch's SDPA on the GPU in float64)."""
    q, K, V, lens_t = _case(2, 32, 8, 600, [600, 600], torch.bfloat16, seed=12)
    ev = _run_step(H, q, K, V, lens_t, [600, 600], 600, ATTN)
    Ke = torch.repeat_interleave(K.double(), 4, dim=1)
    Ve = torch.repeat_interleave(V.double(), 4, dim=1)
    ref = torch.nn.functional.scaled_dot_product_attention(q.double().unsqueeze(2), Ke, Ve).squeeze(2)
    check_attn(ev.out.cpu().numpy(), ref.cpu().numpy())


# ------------------------------------------------------------ workloads
def _workload_step(H, oracle_mod, w, layer, step, mode, with_attn=True):
    K, V = inputs.layer_cache(w, layer, device="cuda")
    q = inputs.step_query(w, layer, step, device="cuda")
    lens, k = w.lens_at(step), w.budget_at(step)
    ev = _run_step(H, q, K, V, torch.tensor(lens, dtype=torch.int32, device="cuda"), k, w.max_k, mode,
                   with_attn=with_attn)
    qc, Kc, Vc = q.cpu(), K.cpu(), V.cpu()
    ref = oracle_mod.evict_step(mode, qc, Kc, Vc, lens, k, w.max_k, with_attn=False)
    check_scores(ev.scores.cpu().numpy(), ref["s"], lens, what=f"{w.name} L{layer} t{step}")
    n_exact = check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), ref["s"], lens, k, w.max_k,
                              what=f"{w.name} L{layer} t{step}")
    if with_attn:
        out_ref = oracle_mod.sparse_attn(qc, Kc, Vc, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
        check_attn(ev.out.cpu().numpy(), out_ref, what=f"{w.name} L{layer} t{step}")
    return ev, ref, n_exact


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_workload1_planted_heavy_hitters(H, oracle_mod, mode):
    """Full size: 1 layer, B=1, 32 heads, 4096 tokens, 64 planted keys, k=819."""
    w = inputs.config(1)
    ev, ref, n_exact = _workload_step(H, oracle_mod, w, 0, 0, mode)
    K, _ = inputs.layer_cache(w, 0, device="cuda")
    q = inputs.step_query(w, 0, 0, device="cuda")
    proj = torch.einsum("hjd,hd->hj", K[0].float(), torch.nn.functional.normalize(q[0].float(), dim=-1))
    planted = torch.where((proj > 2 * 128 ** 0.5).all(0))[0].cpu().tolist()
    assert len(planted) == 64
    assert set(planted) <= set(ev.idx[0, :819].cpu().tolist())


@pytest.mark.parametrize("layer,step", [(0, 0), (31, 63)])
def test_workload2_full_size_sampled(H, oracle_mod, layer, step):
    """Full size, the benchmark's workload: B=8, 32 heads MHA, 4096+step tokens, k=20 %."""
    w = inputs.config(2)
    _workload_step(H, oracle_mod, w, layer, step, ATTN)


def test_workload3_ragged_32k_sampled(H, oracle_mod):
    w = inputs.config(3)
    _workload_step(H, oracle_mod, w, 0, 31, ATTN)


def test_workload4_gqa_128k_sampled(H, oracle_mod):
    w = inputs.config(4)
    _workload_step(H, oracle_mod, w, 5, 7, ATTN)


def test_workload5_accumulating_sweep_reduced(H, oracle_mod):
    """The budget sweep with cumulative importance, one sequence at 8K tokens
    over several steps, budgets 5 % and 50 %."""
    for frac in (0.05, 0.5):
        w = inputs.config(5, batch=1, layers=1, prompt_lens=(8192,), steps=3, budget_frac=frac)
        K, V = inputs.layer_cache(w, 0)
        Kd, Vd = K.cuda(), V.cuda()
        A = torch.zeros(1, w.capacity, device="cuda")
        A_ref = np.zeros((1, w.capacity))
        for t in range(w.steps):
            lens, k = w.lens_at(t), w.budget_at(t)
            q = inputs.step_query(w, 0, t)
            ev = _run_step(H, q.cuda(), Kd, Vd, torch.tensor(lens, dtype=torch.int32, device="cuda"), k,
                           w.max_k, ATTN, accum=A)
            r = oracle_mod.evict_step(ATTN, q, K, V, lens, k, w.max_k, accum=A_ref, with_attn=False)
            A_ref = r["accum"]
            check_scores(A.cpu().numpy(), A_ref, lens, what=f"accum {frac} t{t}")
            check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), A_ref, lens, k, w.max_k)

"""GPU parity of the split step (hill_evict_step_begin / hill_evict_step_end),
the building block of the layer-pipelined evaluation (Sec. 4.3):

* the selection of end() alone (RAW mode: end() selects on the caller's
  scores, building the leading-digit histogram itself) against the oracle's
  sort of the same keys, bit for bit: cluster sizes 1 to 8, heavy exact ties,
  signed zeros, flat key distributions with large crossing buckets, BKP
  windows and hit tables, and the budget edge cases;
* the split step against the oracle (scores, selection by the gap rule) and
  against the fused hill_evict_step (RAW: bit for bit; ATTN: scores within
  the tolerance, since the split step's scoring grid -- 17/20 of the SMs --
  combines the softmax partials in another order), from the 16-bit
  keys and from their E4M3 shadow (begin_f8 against hill_evict_step_f8);
* two streams and rotating workspaces over the layers of the 32K and 128K
  workloads, eagerly and in a CUDA graph, bit for bit against the same split
  calls issued one after another on one stream, and within the tolerance of
  the serial fused step.
"""
import numpy as np
import pytest
import torch

from paper_2602_18750_gb300 import inputs
from parity_util import check_scores, check_selection

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


def _end_select(H, s, lens, k, max_k, recent=0, hits=None):
    """end() in RAW mode: the selection on the caller's keys s [B][cap]."""
    B, cap = s.shape
    q = torch.zeros(B, 4, 128, dtype=torch.float16, device="cuda")
    K = torch.zeros(B, 4, 8, 128, dtype=torch.float16, device="cuda")
    desc = H.make_desc(q, K)
    desc.capacity = cap
    ws = H.alloc_workspace(desc, RAW, max_k)
    idx = torch.full((B, max_k), -5, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -5, dtype=torch.int32, device="cuda")
    H.hill_evict_step_end(desc, _i32(lens), _i32(k), max_k, RAW, None, s.cuda(), idx, cnt, ws, recent=recent,
                          hits=hits)
    return idx, cnt


def _keys(kind, B, cap, seed):
    g = torch.Generator().manual_seed(seed)
    if kind == "lognormal":            # few keys in the crossing bucket: gathered candidates
        return torch.exp(torch.randn(B, cap, generator=g) * 4)
    if kind == "uniform":              # one octave: a large crossing bucket, cluster histograms
        return 1.0 + torch.rand(B, cap, generator=g)
    if kind == "ties":                 # heavy exact ties and signed zeros
        s = torch.randint(-3, 4, (B, cap), generator=g).float()
        s[:, ::5] = -0.0
        return s
    if kind == "softmaxlike":          # sums of softmax weights: small positive values
        return torch.rand(B, cap, generator=g) ** 6 * 1e-3
    raise ValueError(kind)


@pytest.mark.parametrize("kind", ["lognormal", "uniform", "ties", "softmaxlike"])
@pytest.mark.parametrize("cap", [700, 4096, 5000, 12000, 40000, 131079])
def test_end_select_matches_oracle(H, oracle_mod, kind, cap):
    """One CTA and clusters of 2, 4 and 8 CTAs per row; budgets from one
    token to most of the sequence."""
    B = 3
    s = _keys(kind, B, cap, cap + len(kind))
    lens = [cap, cap - 37, max(1, cap // 3)]
    k = [max(1, cap // 10), 1, lens[2] - 1]
    max_k = max(k) + 3
    idx, cnt = _end_select(H, s, lens, k, max_k)
    H.hill_sync_status()
    idx_o, cnt_o, _ = oracle_mod.topk(s.numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(cnt.cpu().numpy(), cnt_o)
    assert np.array_equal(idx.cpu().numpy(), idx_o)


def test_end_select_budget_edges(H, oracle_mod):
    """k = 0, k = len, k > len, empty and one-token sequences, and a budget
    above max_k (count capped, device error word raised)."""
    cap = 9000
    s = _keys("lognormal", 5, cap, 3)
    lens = [cap, 0, 1, 5000, 8000]
    k = [0, 4, 1, 5000, 9999]
    idx, cnt = _end_select(H, s, lens, k, 9000)
    H.hill_sync_status()
    idx_o, cnt_o, _ = oracle_mod.topk(s.numpy().astype(np.float64), lens, k, 9000)
    assert np.array_equal(cnt.cpu().numpy(), cnt_o) and np.array_equal(idx.cpu().numpy(), idx_o)
    idx, cnt = _end_select(H, s, [cap] * 5, [100, 20, 30, 40, 50], 32)
    with pytest.raises(H.HillError) as ei:
        H.hill_sync_status()
    assert ei.value.status == H.HILL_ERR_DEVICE
    assert cnt.cpu().tolist() == [32, 20, 30, 32, 32]
    H.hill_sync_status()


@pytest.mark.parametrize("recent", [0, 37, 4000])
@pytest.mark.parametrize("cap", [3000, 40000])
def test_end_select_bkp_window_and_hits(H, oracle_mod, recent, cap):
    """The pinned window and the hit-rate table (Sec. 4.2) of end()'s
    selection equal the oracle's BKP selection over three steps."""
    B = 2
    lens = [cap, cap // 2 + 11]
    k = [cap // 10, cap // 20]
    max_k = max(k) + recent
    hits = torch.zeros(B, cap, dtype=torch.int16, device="cuda")
    hits_ref = np.zeros((B, cap), dtype=np.uint16)
    for step in range(3):
        s = _keys("lognormal", B, cap, 100 * step + cap)
        idx, cnt = _end_select(H, s, lens, k, max_k, recent=recent, hits=hits)
        H.hill_sync_status()
        idx_o, cnt_o, _, hits_ref = oracle_mod.bkp_select(s.numpy().astype(np.float64), lens, k, recent, max_k,
                                                          hits_ref)
        assert np.array_equal(cnt.cpu().numpy(), cnt_o)
        assert np.array_equal(idx.cpu().numpy(), idx_o)
        assert np.array_equal(hits.cpu().numpy().view(np.uint16), hits_ref)


SHAPES = [
    # B, H, Hkv, cap, lens, k
    (3, 8, 8, 1000, [1000, 517, 33], [200, 103, 40]),
    (2, 32, 8, 700, [700, 1], [64, 5]),
    (2, 8, 1, 300, [300, 299], [30, 299]),
    (4, 4, 2, 129, [129, 0, 64, 95], [13, 3, 64, 0]),
    (2, 32, 1, 700, [700, 333], [70, 33]),
    (2, 40, 40, 300, [300, 130], [60, 26]),
    (2, 8, 8, 40000, [40000, 23457], [4000, 2345]),
]


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_split_step_matches_oracle_and_fused(H, oracle_mod, mode, shape):
    B, Hq, Hkv, cap, lens, k = shape
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=cap + Hq,
                                         kind="zipf" if Hq == Hkv else "normal")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    max_k = max(max(k), 1)
    desc = H.make_desc(q, K, V)
    ws = H.alloc_workspace(desc, mode, max_k)
    scores = torch.full((B, cap), float("nan"), device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_evict_step_begin(desc, q, K, lens_t, max_k, mode, None, scores, ws)
    H.hill_evict_step_end(desc, lens_t, _i32(k), max_k, mode, None, scores, idx, cnt, ws)
    H.hill_sync_status()
    ref = oracle_mod.evict_step(mode, q.cpu(), K.cpu(), V.cpu(), lens, k, max_k, with_attn=False)
    check_scores(scores.cpu().numpy(), ref["s"], lens)
    check_selection(idx.cpu().numpy(), cnt.cpu().numpy(), ref["s"], lens, k, max_k)
    # the selection is exact on its own keys
    idx_o, cnt_o, _ = oracle_mod.topk(scores.cpu().numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)
    # the fused step: RAW sums do not depend on the grid (bit-identical
    # scores and selection); ATTN scores agree within the tolerance
    ev = H.Evictor(q, K, V, max_k, mode=mode, with_attn=False)
    ev.step(q, K, V, lens_t, _i32(k))
    H.hill_sync_status()
    check_scores(scores.cpu().numpy(), ev.scores.cpu().numpy().astype(np.float64), lens, what="split vs fused")
    if mode == RAW:
        for b, n in enumerate(lens):
            assert torch.equal(scores[b, :n], ev.scores[b, :n])
        assert torch.equal(idx, ev.idx) and torch.equal(cnt, ev.count)


@pytest.mark.parametrize("mode", [ATTN, RAW])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"B{s[0]}H{s[1]}kv{s[2]}cap{s[3]}")
def test_split_step_f8_matches_oracle_and_fused(H, oracle_mod, mode, shape):
    """hill_evict_step_begin_f8 + end on the E4M3 shadow: scores against the
    oracle's logits on the 8-bit operands, the selection exact on its own
    keys, and against the fused hill_evict_step_f8 (RAW bit for bit, ATTN
    within the tolerance)."""
    B, Hq, Hkv, cap, lens, k = shape
    q, K, V, lens_t = inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.bfloat16, seed=cap + 3 * Hq,
                                         kind="zipf" if Hq == Hkv else "normal")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    max_k = max(max(k), 1)
    desc = H.make_desc(q, K, V)
    k8, ks = H.alloc_shadow(desc)
    H.hill_quantize_k(desc, K, _i32([0] * B), lens_t, cap, k8, ks)
    ws = H.alloc_workspace(desc, mode, max_k)
    scores = torch.full((B, cap), float("nan"), device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    H.hill_evict_step_begin_f8(desc, q, k8, ks, lens_t, max_k, mode, None, scores, ws)
    H.hill_evict_step_end(desc, lens_t, _i32(k), max_k, mode, None, scores, idx, cnt, ws)
    H.hill_sync_status()
    codes, scale = oracle_mod.quantize_rows(K.cpu())
    s_ref = oracle_mod.scores(mode, oracle_mod.logits_q8(q.cpu(), codes, scale, lens), lens)
    check_scores(scores.cpu().numpy(), s_ref, lens)
    check_selection(idx.cpu().numpy(), cnt.cpu().numpy(), s_ref, lens, k, max_k)
    idx_o, cnt_o, _ = oracle_mod.topk(scores.cpu().numpy().astype(np.float64), lens, k, max_k)
    assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)
    s_f = torch.full((B, cap), float("nan"), device="cuda")
    idx_f = torch.empty_like(idx)
    cnt_f = torch.empty_like(cnt)
    H.hill_evict_step_f8(desc, q, k8, ks, K, V, lens_t, _i32(k), max_k, mode, None, s_f, idx_f, cnt_f, None, ws)
    H.hill_sync_status()
    check_scores(scores.cpu().numpy(), s_f.cpu().numpy().astype(np.float64), lens, what="split vs fused")
    if mode == RAW:
        for b, n in enumerate(lens):
            assert torch.equal(scores[b, :n], s_f[b, :n])
        assert torch.equal(idx, idx_f) and torch.equal(cnt, cnt_f)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_split_step_accumulates(H, oracle_mod, mode):
    """Running importance through the split step over three steps."""
    w = inputs.config(5, layers=1, batch=3, prompt_lens=(3000, 1800, 640), steps=3)
    K, V = inputs.layer_cache(w, 0)
    Kd, Vd = K.cuda(), V.cuda()
    q0 = inputs.step_query(w, 0, 0).cuda()
    desc = H.make_desc(q0, Kd, Vd)
    ws = H.alloc_workspace(desc, mode, w.max_k)
    A = torch.zeros(w.batch, w.capacity, device="cuda")
    A_ref = np.zeros((w.batch, w.capacity))
    s = torch.empty(w.batch, w.capacity, device="cuda")
    idx = torch.empty(w.batch, w.max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(w.batch, dtype=torch.int32, device="cuda")
    for t in range(w.steps):
        lens, k = w.lens_at(t), w.budget_at(t)
        q = inputs.step_query(w, 0, t)
        H.hill_evict_step_begin(desc, q.cuda(), Kd, _i32(lens), w.max_k, mode, A, s, ws)
        H.hill_evict_step_end(desc, _i32(lens), _i32(k), w.max_k, mode, A, s, idx, cnt, ws)
        H.hill_sync_status()
        r = oracle_mod.evict_step(mode, q, K, V, lens, k, w.max_k, accum=A_ref, with_attn=False)
        A_ref = r["accum"]
        check_scores(A.cpu().numpy(), A_ref, lens, what=f"accum step {t}")
        check_selection(idx.cpu().numpy(), cnt.cpu().numpy(), A_ref, lens, k, w.max_k)
        idx_o, cnt_o, _ = oracle_mod.topk(A.cpu().numpy().astype(np.float64), lens, k, w.max_k)
        assert np.array_equal(idx.cpu().numpy(), idx_o) and np.array_equal(cnt.cpu().numpy(), cnt_o)


def test_split_step_bkp_window_and_hits(H, oracle_mod):
    """end() with a window and a hit table (Sec. 4.2): over two steps, the
    kept set and the table equal the oracle's BKP selection on the step's own
    scores, and the scores stay within the tolerance of the oracle's."""
    B, Hq, cap = 2, 8, 40000
    lens, k, recent = [40000, 30001], [3000, 2000], 128
    q, K, V, lens_t = inputs.random_case(B, Hq, Hq, 128, cap, lens, seed=71, kind="zipf")
    q, K, V, lens_t = q.cuda(), K.cuda(), V.cuda(), lens_t.cuda()
    max_k = max(k) + recent
    desc = H.make_desc(q, K, V)
    ws = H.alloc_workspace(desc, ATTN, max_k)
    hits = torch.zeros(B, cap, dtype=torch.int16, device="cuda")
    hits_ref = np.zeros((B, cap), dtype=np.uint16)
    s = torch.empty(B, cap, device="cuda")
    idx = torch.empty(B, max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(B, dtype=torch.int32, device="cuda")
    ref = oracle_mod.evict_step(ATTN, q.cpu(), K.cpu(), V.cpu(), lens, k, max_k, with_attn=False)
    for _ in range(2):
        H.hill_evict_step_begin(desc, q, K, lens_t, max_k, ATTN, None, s, ws)
        H.hill_evict_step_end(desc, lens_t, _i32(k), max_k, ATTN, None, s, idx, cnt, ws, recent=recent, hits=hits)
        H.hill_sync_status()
        check_scores(s.cpu().numpy(), ref["s"], lens)
        idx_o, cnt_o, _, hits_ref = oracle_mod.bkp_select(s.cpu().numpy().astype(np.float64), lens, k, recent,
                                                          max_k, hits_ref)
        assert np.array_equal(cnt.cpu().numpy(), cnt_o) and np.array_equal(idx.cpu().numpy(), idx_o)
        assert np.array_equal(hits.cpu().numpy().view(np.uint16), hits_ref)


def _pipelined_layers(H, w, layers, mode, form, graph=False, nws=3):
    """Evaluation + selection of `layers` layers at the last decode step, in
    one of three forms: "fused" (one hill_evict_step per layer), "split" (begin
    then end per layer on one stream), "piped" (begin on one stream, end on a
    second, nws rotating workspaces: end of layer l before begin of layer
    l + nws)."""
    t = w.steps - 1
    lens_t, k_t = _i32(w.lens_at(t)), _i32(w.budget_at(t))
    caches = [inputs.layer_cache(w, l, device="cuda") for l in range(layers)]
    qs = [inputs.step_query(w, l, t, device="cuda") for l in range(layers)]
    desc = H.make_desc(qs[0], caches[0][0], caches[0][1])
    ws = [H.alloc_workspace(desc, mode, w.max_k) for _ in range(nws)]
    scores = torch.empty(layers, w.batch, w.capacity, device="cuda")
    idx = torch.empty(layers, w.batch, w.max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(layers, w.batch, dtype=torch.int32, device="cuda")
    main = torch.cuda.Stream()
    side = torch.cuda.Stream()
    torch.cuda.synchronize()   # the inputs were made on the default stream

    def issue():
        if form == "fused":
            for l in range(layers):
                K, V = caches[l]
                H.hill_evict_step(desc, qs[l], K, V, lens_t, k_t, w.max_k, mode, None, scores[l], idx[l], cnt[l],
                                  None, ws[0], main)
        elif form == "split":
            for l in range(layers):
                H.hill_evict_step_begin(desc, qs[l], caches[l][0], lens_t, w.max_k, mode, None, scores[l], ws[0], main)
                H.hill_evict_step_end(desc, lens_t, k_t, w.max_k, mode, None, scores[l], idx[l], cnt[l], ws[0],
                                      stream=main)
        else:
            done = [torch.cuda.Event() for _ in range(layers)]
            for l in range(layers):
                if l >= nws:
                    main.wait_event(done[l - nws])
                K, V = caches[l]
                H.hill_evict_step_begin(desc, qs[l], K, lens_t, w.max_k, mode, None, scores[l], ws[l % nws], main)
                ev = torch.cuda.Event()
                ev.record(main)
                side.wait_event(ev)
                H.hill_evict_step_end(desc, lens_t, k_t, w.max_k, mode, None, scores[l], idx[l], cnt[l],
                                      ws[l % nws], stream=side)
                done[l].record(side)
            main.wait_event(done[-1])

    if graph:   # captured once, replayed twice (as the benchmark runs it)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=main):
            issue()
        with torch.cuda.stream(main):
            g.replay()
            g.replay()
    else:
        with torch.cuda.stream(main):
            issue()
    main.synchronize()
    H.hill_sync_status(main)
    return scores, idx, cnt


@pytest.mark.parametrize("n,mode", [(3, ATTN), (4, ATTN), (4, RAW)])
def test_two_stream_pipeline_full_size(H, oracle_mod, n, mode):
    """Five layers of the 32K ragged (B 4) and 128K GQA (B 1) workloads: the
    pipelined begin / end on two streams (two and three rotating workspaces
    and one per layer, eagerly and captured in a CUDA graph) gives the split calls' scores and
    selections bit for bit; those agree with the serial fused step within
    the tolerance, and its selections are exact on their own keys."""
    w = inputs.config(n)
    layers = 5
    lens, k = w.lens_at(w.steps - 1), w.budget_at(w.steps - 1)
    a = _pipelined_layers(H, w, layers, mode, "split")
    for graph in (False, True):
        for nws in (2, 3, layers):
            b = _pipelined_layers(H, w, layers, mode, "piped", graph, nws)
            for l in range(layers):
                for bb, m in enumerate(lens):
                    assert torch.equal(a[0][l, bb, :m], b[0][l, bb, :m]), f"scores layer {l} seq {bb}"
            assert torch.equal(a[1], b[1]) and torch.equal(a[2], b[2])
    f = _pipelined_layers(H, w, layers, mode, "fused")
    for l in range(layers):
        check_scores(a[0][l].cpu().numpy(), f[0][l].cpu().numpy().astype(np.float64), lens, what=f"layer {l}")
        idx_o, cnt_o, _ = oracle_mod.topk(a[0][l].cpu().numpy().astype(np.float64), lens, k, w.max_k)
        assert np.array_equal(a[1][l].cpu().numpy(), idx_o) and np.array_equal(a[2][l].cpu().numpy(), cnt_o)

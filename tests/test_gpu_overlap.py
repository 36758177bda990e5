"""The layer-pipelined schedule (the APP analogue, Sec. 4.3): evaluation and
selection of layer l + 1 on one stream while the sparse attention of layer l
runs on a second stream, ordered only by an event after each selection.  The
results must be bit-identical to the serial schedule, eagerly and when the
two-stream schedule is captured in one CUDA graph.
"""
import pytest
import torch

from paper_2602_18750_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2602_18750_gb300 import build, hill
    build.build()
    hill.load()
    return hill


def test_pipelined_layers_equal_serial(H):
    L, B, Hq, Hkv, cap = 4, 3, 16, 4, 900
    lens, k = [900, 640, 77], [180, 128, 15]
    max_k = 180
    layers = [inputs.random_case(B, Hq, Hkv, 128, cap, lens, dtype=torch.float16, seed=70 + l, kind="zipf")
              for l in range(L)]
    layers = [tuple(x.cuda() for x in c) for c in layers]
    lens_t = layers[0][3]
    k_t = torch.tensor(k, dtype=torch.int32, device="cuda")
    desc = H.make_desc(layers[0][0], layers[0][1], layers[0][2])
    ws = [H.alloc_workspace(desc, 0, max_k) for _ in range(2)]

    def buffers():
        return ([torch.empty(B, max_k, dtype=torch.int32, device="cuda") for _ in range(L)],
                [torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(L)],
                [torch.empty(B, Hq, 128, device="cuda") for _ in range(L)])

    # serial: one fused step per layer
    idx0, cnt0, out0 = buffers()
    for l, (q, K, V, _) in enumerate(layers):
        H.hill_evict_step(desc, q, K, V, lens_t, k_t, max_k, 0, None, None, idx0[l], cnt0[l], out0[l], ws[0])
    H.hill_sync_status()

    main = torch.cuda.Stream()
    side = torch.cuda.Stream()

    def pipelined(idx, cnt, out):
        fork = torch.cuda.Event()
        fork.record(main)
        side.wait_event(fork)
        for l, (q, K, V, _) in enumerate(layers):
            H.hill_evict_step(desc, q, K, V, lens_t, k_t, max_k, 0, None, None, idx[l], cnt[l], None, ws[0], main)
            sel = torch.cuda.Event()
            sel.record(main)
            side.wait_event(sel)
            H.hill_gather_sparse_attn(desc, q, K, V, idx[l], cnt[l], max_k, out[l], ws[1], side)
        join = torch.cuda.Event()
        join.record(side)
        main.wait_event(join)

    idx1, cnt1, out1 = buffers()
    with torch.cuda.stream(main):
        pipelined(idx1, cnt1, out1)
    main.synchronize()
    H.hill_sync_status()
    idx2, cnt2, out2 = buffers()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=main):
        pipelined(idx2, cnt2, out2)
    g.replay()
    torch.cuda.synchronize()
    H.hill_sync_status()
    for l in range(L):
        for got in ((idx1, cnt1, out1), (idx2, cnt2, out2)):
            assert torch.equal(got[0][l], idx0[l]) and torch.equal(got[1][l], cnt0[l])
            assert torch.equal(got[2][l], out0[l])


@pytest.mark.parametrize("wl", [2, 4])
def test_pipelined_full_size_equals_serial(H, wl):
    """The benchmark's default schedule at full per-layer size (4K MHA and
    128K GQA workloads, three layers, last decode step, in a CUDA graph as
    the benchmark runs it) gives the serial step's selection and attention
    bit for bit; the serial step itself is checked against the oracle by the
    sampled full-size parity tests."""
    w = inputs.config(wl)
    L = 3
    t = w.steps - 1
    cache = [inputs.layer_cache(w, l, device="cuda") for l in range(L)]
    qs = [inputs.step_query(w, l, t, device="cuda") for l in range(L)]
    lens_t = torch.tensor(w.lens_at(t), dtype=torch.int32, device="cuda")
    k_t = torch.tensor(w.budget_at(t), dtype=torch.int32, device="cuda")
    desc = H.make_desc(qs[0], cache[0][0], cache[0][1])
    ws = [H.alloc_workspace(desc, 0, w.max_k) for _ in range(2)]
    B, Hq = qs[0].shape[0], qs[0].shape[1]

    def buffers():
        return ([torch.empty(B, w.max_k, dtype=torch.int32, device="cuda") for _ in range(L)],
                [torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(L)],
                [torch.empty(B, Hq, 128, device="cuda") for _ in range(L)])

    idx0, cnt0, out0 = buffers()
    for l in range(L):
        H.hill_evict_step(desc, qs[l], cache[l][0], cache[l][1], lens_t, k_t, w.max_k, 0, None, None, idx0[l],
                          cnt0[l], out0[l], ws[0])
    H.hill_sync_status()
    main, side = torch.cuda.Stream(), torch.cuda.Stream()
    idx1, cnt1, out1 = buffers()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=main):
        fork = torch.cuda.Event()
        fork.record(main)
        side.wait_event(fork)
        for l in range(L):
            H.hill_evict_step(desc, qs[l], cache[l][0], cache[l][1], lens_t, k_t, w.max_k, 0, None, None,
                              idx1[l], cnt1[l], None, ws[0], main)
            sel = torch.cuda.Event()
            sel.record(main)
            side.wait_event(sel)
            H.hill_gather_sparse_attn(desc, qs[l], cache[l][0], cache[l][1], idx1[l], cnt1[l], w.max_k, out1[l],
                                      ws[1], side)
        join = torch.cuda.Event()
        join.record(side)
        main.wait_event(join)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    H.hill_sync_status()
    for l in range(L):
        assert torch.equal(idx1[l], idx0[l]) and torch.equal(cnt1[l], cnt0[l])
        assert torch.equal(out1[l], out0[l])

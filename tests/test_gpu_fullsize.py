"""GPU parity at the benchmark's full sizes, through the same hill_evict_step
launch path that bench.py times, against the CPU oracle on the same seeded
inputs (one sampled layer, every sequence, every token):

* the accumulating sweep at its benchmark point (B 8 x 64K tokens, 32 heads
  MHA, k = 20 %), cumulative importance carried over three decode steps;
* the sweep's widest batch at 8K tokens (B 16) at the smallest and largest
  budgets (5 % and 50 %), accumulating;
* RAW importance (Sec. 4.4) on the 32K ragged and the 128K GQA workloads;
* asymmetric-precision scoring (Sec. 4.4, E4M3 key shadow) on one full layer
  of the 32K ragged workload, scores and selection.

Scores are compared token by token (1e-3 relative), selections with the
boundary-gap rule, attention outputs within 2e-3 absolute on the GPU's own
index set.
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


def _accumulating_steps(H, oracle_mod, w, layer, steps, mode=ATTN):
    """Decode steps 0 .. steps-1 of one layer of w with the running importance
    carried across them, as the benchmark runs it: every step checks this
    step's scores, the running sums and the selection made on them; the last
    step also checks the sparse attention."""
    K, V = inputs.layer_cache(w, layer, device="cuda")
    Kc, Vc = K.cpu(), V.cpu()
    ev = H.Evictor(inputs.step_query(w, layer, 0, device="cuda"), K, V, w.max_k, mode=mode)
    A = torch.zeros(w.batch, w.capacity, device="cuda")
    A_ref = np.zeros((w.batch, w.capacity))
    for t in range(steps):
        lens, k = w.lens_at(t), w.budget_at(t)
        q = inputs.step_query(w, layer, t, device="cuda")
        ev.step(q, K, V, _i32(lens), _i32(k), accum=A)
        H.hill_sync_status()
        qc = q.cpu()
        r = oracle_mod.evict_step(mode, qc, Kc, Vc, lens, k, w.max_k, accum=A_ref, with_attn=False)
        A_ref = r["accum"]
        what = f"{w.name} L{layer} t{t}"
        check_scores(ev.scores.cpu().numpy(), r["s"], lens, what=f"scores {what}")
        check_scores(A.cpu().numpy(), A_ref, lens, what=f"accum {what}")
        check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), A_ref, lens, k, w.max_k, what=what)
    out_ref = oracle_mod.sparse_attn(qc, Kc, Vc, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
    check_attn(ev.out.cpu().numpy(), out_ref, what=f"{w.name} L{layer} t{steps - 1}")


def test_sweep_benchmark_point_b8_64k_accumulating(H, oracle_mod):
    """The sweep point the benchmark runs: B 8 x 65536 tokens, k = 20 %,
    cumulative importance over three decode steps (layer 17)."""
    w = inputs.config(5)
    assert (w.batch, w.prompt_lens[0], w.budget_frac, w.accumulate) == (8, 65536, 0.2, True)
    _accumulating_steps(H, oracle_mod, w, 17, 3)


@pytest.mark.parametrize("frac", [0.05, 0.5])
def test_sweep_b16_8k_accumulating(H, oracle_mod, frac):
    """The sweep's widest batch (16 sequences of 8192 tokens) at its smallest
    and largest budgets, accumulating over three steps."""
    w = inputs.sweep_point(16, 8192, frac)
    _accumulating_steps(H, oracle_mod, w, 3, 3)


def _single_step(H, oracle_mod, w, layer, step, mode):
    K, V = inputs.layer_cache(w, layer, device="cuda")
    q = inputs.step_query(w, layer, step, device="cuda")
    lens, k = w.lens_at(step), w.budget_at(step)
    ev = H.Evictor(q, K, V, w.max_k, mode=mode)
    ev.step(q, K, V, _i32(lens), _i32(k))
    H.hill_sync_status()
    qc, Kc, Vc = q.cpu(), K.cpu(), V.cpu()
    ref = oracle_mod.evict_step(mode, qc, Kc, Vc, lens, k, w.max_k, with_attn=False)
    what = f"{w.name} L{layer} t{step} mode {mode}"
    check_scores(ev.scores.cpu().numpy(), ref["s"], lens, what=what)
    check_selection(ev.idx.cpu().numpy(), ev.count.cpu().numpy(), ref["s"], lens, k, w.max_k, what=what)
    out_ref = oracle_mod.sparse_attn(qc, Kc, Vc, ev.idx.cpu().numpy(), ev.count.cpu().numpy())
    check_attn(ev.out.cpu().numpy(), out_ref, what=what)


def test_raw_mode_32k_ragged(H, oracle_mod):
    """RAW importance (Sec. 4.4) on the 32K ragged workload (B 4, fp16)."""
    _single_step(H, oracle_mod, inputs.config(3), 9, 20, RAW)


def test_raw_mode_128k_gqa(H, oracle_mod):
    """RAW importance on the 128K GQA workload (B 1, 32 query / 8 KV heads, bf16)."""
    _single_step(H, oracle_mod, inputs.config(4), 30, 3, RAW)


@pytest.mark.parametrize("mode", [ATTN, RAW])
def test_score_f8_full_layer_32k_ragged(H, oracle_mod, mode):
    """hill_quantize_k over one whole layer of the 32K ragged workload, then
    hill_evict_step_f8: scores against the oracle's logits on the 8-bit
    operands, the selection against those scores (gap rule), and the
    attention on the 16-bit keys and values."""
    w = inputs.config(3)
    layer, t = 12, w.steps - 1
    K, V = inputs.layer_cache(w, layer, device="cuda")
    q = inputs.step_query(w, layer, t, device="cuda")
    lens, k = w.lens_at(t), w.budget_at(t)
    desc = H.make_desc(q, K, V)
    k8, ks = H.alloc_shadow(desc)
    H.hill_quantize_k(desc, K, _i32([0] * w.batch), _i32(lens), w.capacity, k8, ks)
    ws = H.alloc_workspace(desc, mode, w.max_k)
    scores = torch.full((w.batch, w.capacity), float("nan"), device="cuda")
    idx = torch.empty(w.batch, w.max_k, dtype=torch.int32, device="cuda")
    cnt = torch.empty(w.batch, dtype=torch.int32, device="cuda")
    out = torch.empty(w.batch, w.heads, w.head_dim, device="cuda")
    H.hill_evict_step_f8(desc, q, k8, ks, K, V, _i32(lens), _i32(k), w.max_k, mode, None, scores, idx, cnt, out,
                         ws)
    H.hill_sync_status()
    Kc = K.cpu()
    codes, scale = oracle_mod.quantize_rows(Kc)
    # the shadow rows the scoring read are the oracle's, bit for bit
    for b, n in enumerate(lens):
        assert np.array_equal(k8[b, :, :n].cpu().numpy(), codes[b, :, :n])
        assert np.array_equal(ks[b, :, :n].cpu().numpy(), scale[b, :, :n])
    s_ref = oracle_mod.scores(mode, oracle_mod.logits_q8(q.cpu(), codes, scale, lens), lens)
    what = f"{w.name} L{layer} t{t} E4M3 mode {mode}"
    check_scores(scores.cpu().numpy(), s_ref, lens, what=what)
    check_selection(idx.cpu().numpy(), cnt.cpu().numpy(), s_ref, lens, k, w.max_k, what=what)
    o_ref = oracle_mod.sparse_attn(q.cpu(), Kc, V.cpu(), idx.cpu().numpy(), cnt.cpu().numpy())
    check_attn(out.cpu().numpy(), o_ref, what=what)

"""Comparison rules shared by the GPU parity tests.

Tolerances (fp32 accumulation on the GPU against the float64 oracle):
* importance scores: |gpu - ref| <= 1e-3 * max(|ref|, mean_j |ref|) per token;
* selected index sets: identical when the oracle's relative gap between the
  k-th and (k+1)-th key exceeds 1e-4; otherwise the same size, every token
  clearly above the boundary present and none clearly below it;
* attention outputs: within 2e-3 absolute, the oracle run on the GPU's own
  index set (so ties at the boundary cannot move the comparison).
"""
import numpy as np

SCORE_RTOL = 1e-3
GAP_RTOL = 1e-4
ATTN_ATOL = 2e-3


def check_scores(got, ref, lens, what="scores"):
    got = np.asarray(got, dtype=np.float64)
    for b, n in enumerate(lens):
        if n == 0:
            continue
        g, r = got[b, :n], ref[b, :n]
        floor = np.abs(r).mean()
        err = np.abs(g - r)
        bound = SCORE_RTOL * np.maximum(np.abs(r), floor)
        bad = np.where(err > bound)[0]
        assert bad.size == 0, (f"{what}[b={b}] {bad.size} tokens out of tolerance; first j={bad[0]} "
                               f"gpu={g[bad[0]]!r} ref={r[bad[0]]!r}")


def check_selection(idx, count, key_ref, lens, k, max_k, what="selection"):
    """GPU (idx, count) against the oracle's keys (float64) with the gap rule."""
    idx = np.asarray(idx)
    count = np.asarray(count)
    exact = 0
    for b, n in enumerate(lens):
        kk = min(max(int(k[b]), 0), n, max_k)
        assert int(count[b]) == kk, f"{what}: count[{b}]={count[b]} want {kk}"
        sel = idx[b, :kk]
        assert np.all(idx[b, kk:max_k] == -1), f"{what}: padding of row {b}"
        assert np.all(np.diff(sel) > 0), f"{what}: row {b} not strictly ascending"
        assert kk == 0 or (sel[0] >= 0 and sel[-1] < n), f"{what}: row {b} index out of range"
        if kk == 0 or kk == n:
            assert sel.tolist() == list(range(n))[:kk]
            exact += 1
            continue
        key = key_ref[b, :n]
        order = np.lexsort((np.arange(n), -key))
        want = np.sort(order[:kk])
        sk, sk1 = key[order[kk - 1]], key[order[kk]]
        gap = (sk - sk1) / abs(sk) if sk != 0 else np.inf
        if gap > GAP_RTOL:
            assert np.array_equal(sel, want), f"{what}: row {b} differs with boundary gap {gap:.3g}"
            exact += 1
        else:
            tol = GAP_RTOL * abs(sk)
            must = set(np.where(key > sk + tol)[0].tolist())
            never = set(np.where(key < sk - tol)[0].tolist())
            s = set(sel.tolist())
            assert must <= s, f"{what}: row {b} misses {sorted(must - s)[:5]}"
            assert not (never & s), f"{what}: row {b} holds {sorted(never & s)[:5]}"
    return exact


def check_attn(got, ref, what="attention"):
    got = np.asarray(got, dtype=np.float64)
    err = np.abs(got - ref)
    worst = np.unravel_index(np.argmax(err), err.shape) if err.size else None
    assert err.size == 0 or err.max() <= ATTN_ATOL, (f"{what}: max abs err {err.max():.3g} at {worst} "
                                                     f"gpu={got[worst]!r} ref={ref[worst]!r}")

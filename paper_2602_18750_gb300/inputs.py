"""Seeded synthetic inputs shaped like HillInfer's workloads (arxiv 2602.18750).

This module only draws inputs: query vectors, key/value caches, per-sequence
lengths and budgets.  It contains none of the evaluation arithmetic (no
scoring, softmax, aggregation, selection or attention) and is the one module
that both the CUDA path's tests/benchmark and the oracle's tests use.

The paper's models and datasets (Qwen-7B, LLaMA, OPT; LongBench, PG-19 and the
LM-eval tasks, Sec. 5.2) are not available, so the caches are synthetic with
the shapes the paper uses (Qwen-7B: 32 layers, 32 heads, head_dim 128; FP16
KV; alpha = 20 %, batch 8, Sec. 5.2) and with a controlled attention skew:

* ``normal``   K, V, q ~ N(0, 1).
* ``planted``  normal, plus P heavy-hitter positions: for each planted token j
               and each KV head g, the component of K[g, j] along the unit
               query direction of the query heads of g is replaced by
               4 * sqrt(d) (its projection becomes 4x a typical key norm).
* ``zipf``     per (layer, sequence, KV head) a fixed direction u ~ N(0, I)
               and a random permutation pi of the prompt positions; prompt key
               j is e_j with its component along u replaced by
               sqrt(d) * t_j / |u|, t_j = -1.1 * ln(pi(j) + 1) centred, so that
               q.K_j / sqrt(d) ~ t_j for q ~ u: attention mass follows a
               Zipf(1.1) law over a random order of the tokens.  The query at a
               step is u + 0.25 * eps.  Tokens appended during decoding
               (positions >= the prompt length) are N(0, 1).
* ``outlier``  normal, plus a fraction of tokens whose whole key vector (all
               KV heads) is scaled by 8.

All draws come from torch generators seeded by (seed, tag, layer, ...), on the
requested device, in float32, then rounded to the cache dtype.
"""
from __future__ import annotations

import dataclasses
import math
import zlib

import torch


def _gen(device, *parts) -> torch.Generator:
    key = zlib.crc32(repr(parts).encode()) & 0x7FFFFFFF
    g = torch.Generator(device=device)
    g.manual_seed(key)
    return g


@dataclasses.dataclass
class Workload:
    """One of the five benchmark workloads (or a scaled-down copy of one)."""
    name: str
    layers: int
    batch: int
    heads: int
    kv_heads: int
    head_dim: int
    prompt_lens: tuple          # per sequence, tokens in the cache at step 0
    steps: int                  # decode steps; step t has prompt_len + t tokens
    dtype: torch.dtype
    kind: str                   # normal | planted | zipf | outlier
    budget_frac: float | None   # k = floor(frac * len)
    budget_tokens: int | None   # or a fixed k
    accumulate: bool = False
    planted: int = 0
    outlier_frac: float = 0.0
    seed: int = 0

    @property
    def capacity(self) -> int:
        return max(self.prompt_lens) + max(self.steps - 1, 0)

    def lens_at(self, step: int) -> list[int]:
        return [p + step for p in self.prompt_lens]

    def budget_at(self, step: int) -> list[int]:
        lens = self.lens_at(step)
        if self.budget_tokens is not None:
            return [self.budget_tokens for _ in lens]
        return [int(math.floor(self.budget_frac * n)) for n in lens]

    @property
    def max_k(self) -> int:
        return max(max(self.budget_at(t)) for t in range(max(self.steps, 1)))

    def kv_bytes(self) -> int:
        el = 2
        return 2 * self.layers * self.batch * self.kv_heads * self.capacity * self.head_dim * el


def config(n: int, *, seed: int = 0, **over) -> Workload:
    """The five workloads (1-based), optionally with fields overridden."""
    if n == 1:
        w = Workload("cfg1-planted-mha-4k", 1, 1, 32, 32, 128, (4096,), 1, torch.float16,
                     "planted", None, 819, planted=64, seed=seed)
    elif n == 2:
        w = Workload("cfg2-qwen7b-b8-4k", 32, 8, 32, 32, 128, (4096,) * 8, 64, torch.float16,
                     "zipf", 0.2, None, seed=seed)
    elif n == 3:
        g = torch.Generator().manual_seed(zlib.crc32(repr(("cfg3-lens", seed)).encode()))
        lens = tuple(int(x) for x in torch.randint(16384, 32769, (4,), generator=g))
        w = Workload("cfg3-qwen7b-b4-32k-ragged", 32, 4, 32, 32, 128, lens, 32, torch.float16,
                     "zipf", 0.1, None, seed=seed)
    elif n == 4:
        w = Workload("cfg4-llama3-8b-gqa-128k", 32, 1, 32, 8, 128, (131072,), 8, torch.bfloat16,
                     "outlier", None, 2048, outlier_frac=0.005, seed=seed)
    elif n == 5:
        w = Workload("cfg5-sweep-b8-64k-k20", 32, 8, 32, 32, 128, (65536,) * 8, 128,
                     torch.float16, "zipf", 0.2, None, accumulate=True, seed=seed)
    else:
        raise ValueError(f"no workload {n}")
    return dataclasses.replace(w, **over) if over else w


SWEEP_BATCHES = (1, 8, 16)
SWEEP_LENS = (8192, 65536)
SWEEP_BUDGETS = (0.05, 0.10, 0.20, 0.50)


def sweep_point(batch: int, prompt_len: int, budget_frac: float, *, seed: int = 0, **over) -> Workload:
    """One point of the budget/batch sweep: the Qwen-7B-shaped stack (32
    layers, 32 heads MHA, head_dim 128, fp16, Zipf(1.1) skew) with `batch`
    sequences of `prompt_len` tokens, budget floor(budget_frac * len), 128
    decode steps with cumulative importance.  The point (8, 65536, 0.2) is
    config(5) itself."""
    name = f"cfg5-sweep-b{batch}-{prompt_len // 1024}k-k{round(budget_frac * 100)}"
    return config(5, seed=seed, name=name, batch=batch, prompt_lens=(prompt_len,) * batch,
                  budget_frac=budget_frac, **over)


def _unit(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True)


def _query_dirs(w: Workload, layer: int, device) -> torch.Tensor:
    """Per (sequence, query head) base query direction u, float32 [B][H][d]."""
    g = _gen(device, w.seed, w.name, "qdir", layer)
    return torch.randn(w.batch, w.heads, w.head_dim, generator=g, device=device)


def layer_cache(w: Workload, layer: int, device="cpu"):
    """(K, V) of one layer, each [B][Hkv][cap][d] in the workload's dtype."""
    B, Hkv, cap, d = w.batch, w.kv_heads, w.capacity, w.head_dim
    G = w.heads // w.kv_heads
    gk = _gen(device, w.seed, w.name, "K", layer)
    gv = _gen(device, w.seed, w.name, "V", layer)
    K = torch.randn(B, Hkv, cap, d, generator=gk, device=device)
    V = torch.randn(B, Hkv, cap, d, generator=gv, device=device)
    if w.kind == "planted":
        gp = _gen(device, w.seed, w.name, "plant", layer)
        u = _query_dirs(w, layer, device)                      # [B][H][d]
        for b in range(B):
            n = w.prompt_lens[b]
            pos = torch.randperm(n, generator=gp, device=device)[: w.planted]
            for g in range(Hkv):
                # one query head of the group defines the planted direction
                qh = _unit(u[b, g * G])
                rows = K[b, g, pos]                            # [P][d]
                proj = rows @ qh
                K[b, g, pos] = rows - proj[:, None] * qh[None, :] + 4.0 * math.sqrt(d) * qh[None, :]
    elif w.kind == "zipf":
        gz = _gen(device, w.seed, w.name, "zipf", layer)
        u = _query_dirs(w, layer, device)
        for b in range(B):
            n = w.prompt_lens[b]
            for g in range(Hkv):
                ug = u[b, g * G]
                uh = _unit(ug)
                perm = torch.randperm(n, generator=gz, device=device).to(torch.float32)
                t = -1.1 * torch.log(perm + 1.0)
                t = t - t.mean()
                rows = K[b, g, :n]
                proj = rows @ uh
                K[b, g, :n] = (rows - proj[:, None] * uh[None, :]
                               + (math.sqrt(d) * t / ug.norm())[:, None] * uh[None, :])
    elif w.kind == "outlier":
        go = _gen(device, w.seed, w.name, "outlier", layer)
        for b in range(B):
            n = w.prompt_lens[b]
            m = int(math.floor(w.outlier_frac * n))
            pos = torch.randperm(n, generator=go, device=device)[:m]
            K[b, :, pos] *= 8.0
    elif w.kind != "normal":
        raise ValueError(w.kind)
    return K.to(w.dtype), V.to(w.dtype)


def step_query(w: Workload, layer: int, step: int, device="cpu") -> torch.Tensor:
    """q [B][H][d] of one layer at one decode step, in the workload's dtype."""
    g = _gen(device, w.seed, w.name, "q", layer, step)
    eps = torch.randn(w.batch, w.heads, w.head_dim, generator=g, device=device)
    if w.kind in ("zipf", "planted"):
        u = _query_dirs(w, layer, device)
        if w.kind == "zipf":
            q = u + 0.25 * eps
        else:
            q = u
    else:
        q = eps
    return q.to(w.dtype)


def random_case(B, H, Hkv, d, cap, lens, dtype=torch.float16, seed=0, device="cpu",
                kind="normal", planted=0, outlier_frac=0.0):
    """A free-form single-layer case for unit tests: (q, K, V, lens int32 tensor).

    The cache has capacity ``cap`` (>= every length); rows at or beyond a
    sequence's length hold N(0, 1) filler that no result may depend on.
    """
    lens = tuple(int(x) for x in lens)
    assert len(lens) == B and all(0 <= n <= cap for n in lens)
    steps = cap - (max(lens) if lens else 0) + 1
    w = Workload(f"case-{kind}", 1, B, H, Hkv, d, lens, steps, dtype, kind, None, 1,
                 planted=planted, outlier_frac=outlier_frac, seed=seed)
    assert w.capacity == cap
    K, V = layer_cache(w, 0, device)
    q = step_query(w, 0, 0, device)
    return q, K, V, torch.tensor(lens, dtype=torch.int32, device=device)

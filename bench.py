#!/usr/bin/env python
"""Benchmark of the per-decode-step token-importance evaluation (HillInfer,
arxiv 2602.18750) on GB300.

One benchmark step is one decode step of the whole stack: for each of the 32
layers, the token-importance evaluation (score every cached key, aggregate per
token over heads, select the top-k per sequence) and the sparse decode
attention over the selection.  The default workload is the long-context one:
the Qwen-7B-shaped stack (32 layers, 32 heads MHA, head_dim 128, fp16) with 4
sequences of 16K-32K cached tokens (ragged, seeded), 32 decode steps, budget
k = floor(0.1 * len), ATTN importance.  Inputs are synthetic (seeded Zipf(1.1)
attention skew) and resident in HBM; every layer's K cache (~800 MB) is larger
than L2 and the 32 layers are distinct, so no L2 flush is needed between
steps.  The same run then times the evaluation + selection alone on the 128K
GQA workload (1 sequence of 131072 tokens, 32 query / 8 KV heads, bf16,
k = 2048), the other context of 32K tokens or more (the `acceptance` key).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  With N > 1 (torchrun, one rank per GPU) every
rank runs its own replica of the workload on its own sequences (weak
scaling); the only collectives are the timing barrier and the max-reduction
of the elapsed time.  ``--impl reference`` times the CPU oracle on the host
cores on the same workload and metric.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2602_18750_gb300 import inputs  # noqa: E402

METRIC = "cached tokens scored+selected/sec"
# keyed by --serial
SCHEDULES = {
    "split": "layer-pipelined (Sec. 4.3): per layer hill_evict_step_begin (K stream) on one stream, "
             "hill_evict_step_end (normalisation + selection) on a second and the sparse attention on a third, "
             "overlapping the K stream of the next layers; one evaluation workspace per layer",
    "attn-overlap": "layer-pipelined (Sec. 4.3): per layer hill_evict_step without attention on one stream, "
                    "the sparse attention on a second stream, overlapping the next layer's evaluation",
    "serial": "serial (one fused hill_evict_step per layer)",
}
UNIT = "tokens/s"
L2_BYTES = 129 * 1024 * 1024


# ---------------------------------------------------------------- distributed helpers
def dist_env():
    """(rank, world, local_rank) from the torchrun environment (1 process if unset)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def replica_seed(base_seed: int, rank: int) -> int:
    """Each rank evaluates its own sequences: a distinct seed per replica."""
    return base_seed + 1000003 * rank


def max_over_ranks(value: float, device=None) -> float:
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(device=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        if device is not None and device.type == "cuda":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ---------------------------------------------------------------- clocks
def smi_device_id(local: int) -> str:
    """The nvidia-smi identifier of CUDA device `local` (its UUID when torch
    exposes it, so that CUDA_VISIBLE_DEVICES remapping cannot point elsewhere)."""
    try:
        u = str(torch.cuda.get_device_properties(local).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            return vis.split(",")[local].strip()
        return str(local)


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons, each stamped on arrival."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str, period_ms: int = 10):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", gpu_id, "-lms", str(period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def wait_first(self, timeout=3.0):
        t0 = time.time()
        while self.proc is not None and not self.samples and time.time() - t0 < timeout:
            time.sleep(0.02)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=2)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0, t1):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        inside = [s for t, s in self.samples if t0 <= t <= t1 + 0.05]
        note = None
        if not inside:   # a very short timed region: take the samples nearest to it
            near = sorted(self.samples, key=lambda ts: abs(ts[0] - (t0 + t1) / 2))[:3]
            inside = [s for _, s in near]
            note = "no sample inside the timed window; nearest samples used"
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(s[0]) for s in inside if num(s[0]) is not None]
        mx = [num(s[1]) for s in inside if num(s[1]) is not None]
        pw = [num(s[2]) for s in inside if num(s[2]) is not None]
        reasons = set()
        for s in inside:
            for name, v in zip(names[1:], s[4:8]):
                if v.strip().lower() == "active":
                    reasons.add(name)
        out = {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
               "power_w_max": max(pw) if pw else None, "reasons": sorted(reasons), "samples": len(inside)}
        if note:
            out["note"] = note
        return out


# ---------------------------------------------------------------- schedules
def pipelined_form(mode: int, accumulate: bool, lres: int) -> str:
    """The layer-pipelined form of a workload (the E4M3 scoring included).
    RAW scoring adds to the running importance inside the K stream, so with
    one resident layer the next layer's stream would race the selection of the
    previous one on the same running sums."""
    if accumulate and mode == 1 and lres < 2:
        return "attn-overlap"
    return "split"


# Evaluation workspaces the split schedule rotates, at most one per layer: with
# one per layer the K stream never waits for a selection inside a decode step
# (measured on the 128K and 32K workloads: 1-3 % faster per layer than three
# rotating workspaces, whose waits also cost the scoring launch its overlap
# with the previous one)
SPLIT_WORKSPACES = 32


def issue_layers(form, L, st, side, att, with_attn, fused, begin, end, attn):
    """Issue one decode step over L layers on stream st and the helper
    streams side and att.  fused(l, with_attn, stream, wi), begin(l, stream,
    wi), end(l, stream, wi) and attn(l, stream, wi) issue the calls of layer l
    with workspace wi of their stage (evaluation: 0 .. SPLIT_WORKSPACES - 1,
    attention: 0 or 1)."""
    if form == "serial":
        for l in range(L):
            fused(l, with_attn, st, 0)
        return
    fork = torch.cuda.Event()
    fork.record(st)
    side.wait_event(fork)
    helpers = [side]
    if form == "split":
        done = [torch.cuda.Event() for _ in range(L)]
        if with_attn:
            att.wait_event(fork)
            helpers.append(att)
        nw = min(SPLIT_WORKSPACES, L)
        for l in range(L):
            if l >= nw:
                st.wait_event(done[l - nw])   # workspace l % nw is free again
            begin(l, st, l % nw)
            streamed = torch.cuda.Event()
            streamed.record(st)
            side.wait_event(streamed)
            end(l, side, l % nw)
            done[l].record(side)
            if with_attn:
                att.wait_event(done[l])
                attn(l, att, l % 2)
    else:
        for l in range(L):
            fused(l, False, st, 0)
            if with_attn:
                sel = torch.cuda.Event()
                sel.record(st)
                side.wait_event(sel)
                attn(l, side, 0)
    for h in helpers:
        join = torch.cuda.Event()
        join.record(h)
        st.wait_event(join)


def capture_steps(S, stream, issue):
    """One CUDA graph per decode step t of issue(t, stream)."""
    graphs = []
    for t in range(S):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            issue(t, stream)
        graphs.append(g)
    return graphs


def time_replays(graphs, order, warmup, stream, dev, clocks_of=None):
    """Replay `warmup` untimed steps, then time exactly the steps of `order`
    with CUDA events on the launching stream between barrier + synchronize
    pairs; with clocks_of (a device index) sample the clocks meanwhile.
    Returns (ms, clock summary or None)."""
    S = len(graphs)
    with torch.cuda.stream(stream):
        for i in range(warmup):
            graphs[i % S].replay()
    stream.synchronize()
    clocks = None
    if clocks_of is not None:
        clocks = ClockSampler(smi_device_id(clocks_of))
        clocks.wait_first()
    barrier(dev)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0 = time.time()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for t in order:
            graphs[t].replay()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    w1 = time.time()
    barrier(dev)
    info = None
    if clocks is not None:
        info = clocks.summary(w0, w1)
        clocks.stop()
    return e0.elapsed_time(e1), info


def eval_summary(ms, tokens, k_bytes_per_token, layer_steps, world, peak, form):
    gbs = tokens * k_bytes_per_token / (ms / 1e3) / 1e9
    return {
        "what": "evaluation + selection without attention (score + aggregate + select), all layers",
        "schedule": SCHEDULES[form],
        "us_per_layer": round(ms * 1e3 / layer_steps, 2),
        "tokens_per_s": round(world * tokens / (ms / 1e3), 1),
        "k_stream_gbs": round(gbs, 1),
        "k_stream_frac_of_measured_hbm": round(gbs / peak, 4),
        "k_stream_frac_of_8tbs": round(gbs / 8000.0, 4),
    }


# ---------------------------------------------------------------- helpers
def source_digest(path: str) -> str:
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def profile_traffic(kernel_key: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current source of the kernel (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    digest = source_digest(os.path.join(ROOT, "paper_2602_18750_gb300", "csrc", "score.cu"))
    for line in open(path):
        m = re.match(r"\s*(\S+)\s+(\S+)\s+src=(\w+)\s+dram_bytes_per_launch=(\d+)", line)
        if m and m.group(1) == kernel_key and m.group(2) == workload and m.group(3) == digest:
            return int(m.group(4))
    return None


def workload_for(n: int, seed: int, layers_resident: int | None, kv_heads: int | None = None):
    w = inputs.config(n, seed=seed)
    if kv_heads:
        # another head layout of the same workload: its query heads over kv_heads KV heads
        if w.heads % kv_heads:
            raise SystemExit(f"--kv-heads {kv_heads} does not divide {w.heads} query heads")
        w = dataclasses.replace(w, kv_heads=kv_heads, name=f"{w.name}-kv{kv_heads}")
    lres = w.layers
    if layers_resident:
        lres = min(lres, layers_resident)
    return w, lres


def describe(w, lres, mode_name):
    lens0, lens1 = w.lens_at(0), w.lens_at(w.steps - 1)
    return {
        "workload": w.name,
        "layers": w.layers, "layers_resident": lres, "batch": w.batch, "heads": w.heads,
        "kv_heads": w.kv_heads, "head_dim": w.head_dim,
        "tokens_first_step": lens0, "tokens_last_step": lens1, "decode_steps": w.steps,
        "budget": (f"floor({w.budget_frac}*len)" if w.budget_tokens is None else w.budget_tokens),
        "kv_dtype": str(w.dtype).replace("torch.", ""), "skew": w.kind, "importance": mode_name,
        "accumulate": w.accumulate,
        "l2": "inputs larger than L2 (each layer's K > 129 MB; consecutive layers distinct), no flush",
    }


# ---------------------------------------------------------------- our implementation
def run_ours(args):
    import torch.distributed as dist

    from paper_2602_18750_gb300 import build as hbuild
    from paper_2602_18750_gb300 import hill

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    hbuild.build()
    hill.load()

    mode = hill.HILL_SCORE_ATTN if args.mode == "attn" else hill.HILL_SCORE_RAW
    w, lres = workload_for(args.workload, replica_seed(args.seed, rank), args.layers_resident, args.kv_heads)
    if args.layers_resident is None:
        # keep as many layers resident as fit in 70 % of the free device memory
        # (the 64K sweep point needs 8.6 GB of K/V per layer); layers beyond
        # that reuse the resident ones cyclically, each larger than L2
        per_layer = 2 * w.batch * w.kv_heads * w.capacity * w.head_dim * torch.finfo(w.dtype).bits // 8
        free = torch.cuda.mem_get_info(dev)[0]
        lres = max(1, min(lres, int(0.7 * free) // per_layer))
    L, S, B, Hq, Hkv, d = w.layers, w.steps, w.batch, w.heads, w.kv_heads, w.head_dim
    cap, max_k = w.capacity, w.max_k
    bkp = args.bkp_recent >= 0
    if bkp:
        max_k += args.bkp_recent   # the pinned window comes on top of the ranked budget

    # ---------------- resident inputs: caches, queries, lengths, budgets
    t_gen = time.time()
    Kall = torch.empty(lres, B, Hkv, cap, d, dtype=w.dtype, device=dev)
    Vall = torch.empty_like(Kall)
    for l in range(lres):
        K, V = inputs.layer_cache(w, l, device=dev)
        Kall[l].copy_(K)
        Vall[l].copy_(V)
        del K, V
    q_all = torch.empty(S, L, B, Hq, d, dtype=w.dtype, device=dev)
    for t in range(S):
        for l in range(L):
            q_all[t, l].copy_(inputs.step_query(w, l, t, device=dev))
    lens_all = torch.tensor([w.lens_at(t) for t in range(S)], dtype=torch.int32, device=dev)
    k_all = torch.tensor([w.budget_at(t) for t in range(S)], dtype=torch.int32, device=dev)
    accum = torch.zeros(lres, B, cap, dtype=torch.float32, device=dev) if w.accumulate else None
    torch.cuda.synchronize()
    t_gen = time.time() - t_gen

    scores = torch.empty(L, B, cap, dtype=torch.float32, device=dev)
    idx = torch.empty(L, B, max_k, dtype=torch.int32, device=dev)
    count = torch.empty(L, B, dtype=torch.int32, device=dev)
    out = torch.empty(L, B, Hq, d, dtype=torch.float32, device=dev)
    desc = hill.make_desc(q_all[0, 0], Kall[0], Vall[0])
    ws = hill.alloc_workspace(desc, mode, max_k, dev)
    stream = torch.cuda.Stream(device=dev)

    hits = torch.zeros(lres, B, cap, dtype=torch.int16, device=dev) if bkp else None
    f8 = args.f8
    if f8:
        # E4M3 shadow of every resident layer's keys (Sec. 4.4), built before
        # timing; every decode step re-quantises its appended token row
        cs, ss = hill.shadow_shape(desc)
        k8_all = torch.zeros((lres,) + cs, dtype=torch.uint8, device=dev)
        ks_all = torch.zeros((lres,) + ss, dtype=torch.float32, device=dev)
        zeros_b = torch.zeros(B, dtype=torch.int32, device=dev)
        cap_b = torch.full((B,), cap, dtype=torch.int32, device=dev)
        for r in range(lres):
            hill.hill_quantize_k(desc, Kall[r], zeros_b, cap_b, cap, k8_all[r], ks_all[r])
        new_row = lens_all - 1
        torch.cuda.synchronize()

    # The calls of one decode step, per layer l (workspace wi: 0 or 1)
    def fused(t, l, with_attn, st, wi):
        r = l % lres
        acc = accum[r] if accum is not None else None
        o = out[l] if with_attn else None
        if f8:
            hill.hill_quantize_k(desc, Kall[r], new_row[t], lens_all[t], 1, k8_all[r], ks_all[r], st)
            hill.hill_evict_step_f8(desc, q_all[t, l], k8_all[r], ks_all[r], Kall[r], Vall[r], lens_all[t], k_all[t],
                                    max_k, mode, acc, scores[l], idx[l], count[l], o, wss[wi], st)
        elif bkp:
            hill.hill_evict_step_bkp(desc, q_all[t, l], Kall[r], Vall[r], lens_all[t], k_all[t], args.bkp_recent,
                                     max_k, mode, acc, scores[l], idx[l], count[l], hits[r], o, wss[wi], st)
        else:
            hill.hill_evict_step(desc, q_all[t, l], Kall[r], Vall[r], lens_all[t], k_all[t], max_k, mode, acc,
                                 scores[l], idx[l], count[l], o, wss[wi], st)

    def begin(t, l, st, wi):
        r = l % lres
        acc = accum[r] if accum is not None else None
        if f8:
            hill.hill_quantize_k(desc, Kall[r], new_row[t], lens_all[t], 1, k8_all[r], ks_all[r], st)
            hill.hill_evict_step_begin_f8(desc, q_all[t, l], k8_all[r], ks_all[r], lens_all[t], max_k, mode, acc,
                                          scores[l], wss[wi], st)
        else:
            hill.hill_evict_step_begin(desc, q_all[t, l], Kall[r], lens_all[t], max_k, mode, acc, scores[l], wss[wi],
                                       st)

    def end(t, l, st, wi):
        r = l % lres
        hill.hill_evict_step_end(desc, lens_all[t], k_all[t], max_k, mode, accum[r] if accum is not None else None,
                                 scores[l], idx[l], count[l], wss[wi], recent=max(args.bkp_recent, 0),
                                 hits=hits[r] if bkp else None, stream=st)

    def attn(t, l, st, wi):
        r = l % lres
        hill.hill_gather_sparse_attn(desc, q_all[t, l], Kall[r], Vall[r], idx[l], count[l], max_k, out[l], wsa[wi],
                                     st)

    side, att = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    wss = [ws] + [hill.alloc_workspace(desc, mode, max_k, dev) for _ in range(SPLIT_WORKSPACES - 1)]   # evaluation
    wsa = [hill.alloc_workspace(desc, mode, max_k, dev) for _ in range(2)]   # attention
    piped = pipelined_form(mode, w.accumulate, lres)
    form = "serial" if args.serial else piped
    other = piped if args.serial else "serial"

    def issue_step(t, st, frm=form, with_attn=True):
        issue_layers(frm, L, st, side, att, with_attn, lambda l, a_, s_, i_: fused(t, l, a_, s_, i_),
                     lambda l, s_, i_: begin(t, l, s_, i_), lambda l, s_, i_: end(t, l, s_, i_),
                     lambda l, s_, i_: attn(t, l, s_, i_))

    # eager warm-up of every kernel shape, then one CUDA graph per decode step
    with torch.cuda.stream(stream):
        issue_step(0, stream)
        issue_step(0, stream, other)
    hill.hill_sync_status(stream)
    n0 = hill.hill_kernel_launches()
    graphs = capture_steps(S, stream, lambda t, st: issue_step(t, st))
    launches = (hill.hill_kernel_launches() - n0) // S   # kernels per decode step (the same for every step)
    if accum is not None:
        accum.zero_()

    tokens_of = [L * sum(w.lens_at(t)) for t in range(S)]
    order = [(args.warmup + i) % S for i in range(args.steps)]
    # bytes of the key stream the scoring reads per token: the 16-bit keys, or
    # with --f8 the E4M3 codes and one float32 scale per row
    k_bytes_per_token = Hkv * (d + 4) if f8 else Hkv * d * 2

    # ---------------- timed region (device-resident inputs)
    ms_local, clock_info = time_replays(graphs, order, args.warmup, stream, dev, clocks_of=local)
    hill.hill_sync_status(stream)
    ms = max_over_ranks(ms_local, dev)
    tokens = sum(tokens_of[t] for t in order)
    value = world * tokens / (ms / 1e3)
    k_gbs = world * tokens * k_bytes_per_token / (ms / 1e3) / 1e9
    gpu_launches = launches * len(order)
    del graphs

    # ---------------- the other schedule, the same steps, timed the same way
    if accum is not None:
        accum.zero_()
    other_graphs = capture_steps(S, stream, lambda t, st: issue_step(t, st, other))
    ms_other = max_over_ranks(time_replays(other_graphs, order, args.warmup, stream, dev)[0], dev)
    hill.hill_sync_status(stream)
    other_schedule = {
        "schedule": SCHEDULES[other],
        "us_per_layer": round(ms_other * 1e3 / (len(order) * L), 2),
        "tokens_per_s": round(world * tokens / (ms_other / 1e3), 1),
    }
    del other_graphs

    # ---------------- evaluation + selection only (no attention): the same steps
    # with out = NULL, in the pipelined form (the K stream of layer l + 1
    # overlaps the normalisation and selection of layer l) and serially, one
    # graph per decode step, timed like the main region
    peak, peak_kind = measured_peaks()
    eval_forms = {}
    for frm in dict.fromkeys([piped, "serial"]):
        if accum is not None:
            accum.zero_()
        eg = capture_steps(S, stream, lambda t, st: issue_step(t, st, frm, with_attn=False))
        ms_e = max_over_ranks(time_replays(eg, order, args.warmup, stream, dev)[0], dev)
        hill.hill_sync_status(stream)
        del eg
        eval_forms[frm] = eval_summary(ms_e, tokens, k_bytes_per_token, len(order) * L, world, peak, frm)
    eval_select = dict(eval_forms[piped])
    if piped != "serial":
        eval_select["serial"] = eval_forms["serial"]

    # ---------------- scoring stage alone, per launch (roofline of the dominant kernels)
    t_s = S - 1
    lens_s = w.lens_at(t_s)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(L)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(L)]
    with torch.cuda.stream(stream):
        for rep in range(2):
            for l in range(L):
                r = l % lres
                if rep == 1:
                    starts[l].record(stream)
                if f8:
                    hill.hill_score_f8(desc, q_all[t_s, l], k8_all[r], ks_all[r], lens_all[t_s], mode, scores[l],
                                       None, ws, stream)
                else:
                    hill.hill_score(desc, q_all[t_s, l], Kall[r], lens_all[t_s], mode, scores[l], None, ws, stream)
                if rep == 1:
                    ends[l].record(stream)
    stream.synchronize()
    score_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / L
    # also the whole fused step of one layer (eval-step time per layer)
    step_us_per_layer = ms_local * 1e3 / (len(order) * L)
    score_tokens = sum(lens_s)
    alg_bytes = score_tokens * (k_bytes_per_token + 4) + B * Hq * d * 2
    peak, peak_kind = measured_peaks()
    achieved = alg_bytes / (score_ms / 1e3) / 1e9
    roofline = {
        "kernel": "hill_score: hill_score_kernel + hill_attn_finalize_kernel" if mode == 0
        else "hill_score: hill_score_kernel",
        "bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
        "frac": round(achieved / peak, 4), "peak_source": peak_kind,
        "traffic": profile_traffic("hill_score_" + args.mode + ("_f8" if f8 else ""), w.name),
        "algorithmic_bytes_per_launch": alg_bytes,
        "bytes_per_token": (f"Hkv*(d+4) + 4 = {k_bytes_per_token + 4}" if f8
                            else f"Hkv*d*2 + 4 = {k_bytes_per_token + 4}"),
        "launch_us": round(score_ms * 1e3, 2),
    }

    # ---------------- end to end through the C ABI with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, w, lres, hill, desc, mode, Kall, Vall, q_all, lens_all, k_all, accum, scores,
                      idx, count, out, wss, wsa, stream, dev, world, side, att, form)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, lres, Kall, Vall, q_all, mode, seconds=args.cpu_seconds)

    # ---------------- the spec acceptance: evaluation + selection at 32K+
    # context, on the headline workload (above) and on the other long-context
    # workloads, each timed alone in this process after the headline's tensors
    # are released
    acceptance = None
    if not args.no_acceptance and not (f8 or bkp):
        acceptance = {"target": "evaluation + selection K stream >= 0.70 of 8 TB/s at >= 32K tokens"}
        if w.name == inputs.config(3).name:
            acceptance["cfg3"] = dict(eval_select, workload=w.name)
        del Kall, Vall, q_all, accum, scores, idx, count, out, ws, wss, wsa
        torch.cuda.empty_cache()
        for n in (3, 4):
            name = inputs.config(n).name
            if n == 4 or w.name != name:
                acceptance[f"cfg{n}"] = eval_select_only(args, n, hill, dev, world, mode)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms / len(order), 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16" if w.dtype == torch.float16 else "bf16",
            "data": "synthetic", "config": dict(describe(w, lres, args.mode),
                                                **({"bkp_recent": args.bkp_recent} if bkp else {}),
                                                **({"scoring": "e4m3 key shadow"} if f8 else {}),
                                                schedule=SCHEDULES[form]),
            "k_stream_gbs": round(k_gbs, 1),
            "k_stream_frac_of_measured_hbm": round(k_gbs / world / peak, 4),
            "k_stream_frac_of_8tbs": round(k_gbs / world / 8000.0, 4),
            "eval_step_us_per_layer": round(step_us_per_layer, 2),
            "other_schedule": other_schedule,
            "eval_select": eval_select,
            "acceptance": acceptance,
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": gpu_launches,
            "clocks": clock_info, "generate_s": round(t_gen, 1),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def measure_workload(args, w, hill, dev, world, mode, full_step=False, layers_resident=None):
    """Evaluation + selection alone (no attention) on workload w with as many
    layers resident as fit (or `layers_resident`), in the layer-pipelined form
    and serially, one CUDA graph per decode step over all layers, timed like
    the main region; the scoring stage (hill_score) per launch; and with
    full_step the pipelined step with the sparse attention.  Accumulating
    workloads carry their running importance across the timed steps."""
    _, _, local = dist_env()
    L, S, B, Hq, Hkv, d = w.layers, w.steps, w.batch, w.heads, w.kv_heads, w.head_dim
    per_layer = 2 * B * Hkv * w.capacity * d * torch.finfo(w.dtype).bits // 8
    lres = max(1, min(L, int(0.7 * torch.cuda.mem_get_info(dev)[0]) // per_layer))
    if layers_resident:
        lres = min(lres, layers_resident)
    t_gen = time.time()
    Kall = torch.empty(lres, B, Hkv, w.capacity, d, dtype=w.dtype, device=dev)
    Vall = torch.empty_like(Kall)
    for l in range(lres):
        K, V = inputs.layer_cache(w, l, device=dev)
        Kall[l].copy_(K)
        Vall[l].copy_(V)
        del K, V
    order = [(args.warmup + i) % S for i in range(args.steps)]
    steps_used = sorted(set(order) | set(i % S for i in range(args.warmup)))
    q_all = {t: torch.stack([inputs.step_query(w, l, t, device=dev) for l in range(L)]) for t in steps_used}
    lens_all = {t: torch.tensor(w.lens_at(t), dtype=torch.int32, device=dev) for t in steps_used}
    k_all = {t: torch.tensor(w.budget_at(t), dtype=torch.int32, device=dev) for t in steps_used}
    accum = torch.zeros(lres, B, w.capacity, dtype=torch.float32, device=dev) if w.accumulate else None
    scores = torch.empty(L, B, w.capacity, dtype=torch.float32, device=dev)
    idx = torch.empty(L, B, w.max_k, dtype=torch.int32, device=dev)
    count = torch.empty(L, B, dtype=torch.int32, device=dev)
    out = torch.empty(L, B, Hq, d, dtype=torch.float32, device=dev) if full_step else None
    desc = hill.make_desc(q_all[steps_used[0]][0], Kall[0], Vall[0])
    wss = [hill.alloc_workspace(desc, mode, w.max_k, dev) for _ in range(SPLIT_WORKSPACES)]
    wsa = [hill.alloc_workspace(desc, mode, w.max_k, dev) for _ in range(2)] if full_step else None
    stream, side, att = (torch.cuda.Stream(device=dev) for _ in range(3))
    torch.cuda.synchronize(dev)   # the inputs were made on the default stream
    t_gen = time.time() - t_gen

    def acc(l):
        return accum[l % lres] if accum is not None else None

    def issue(t, st, frm, with_attn):
        def fused(l, a_, s_, wi):
            hill.hill_evict_step(desc, q_all[t][l], Kall[l % lres], Vall[l % lres], lens_all[t], k_all[t], w.max_k,
                                 mode, acc(l), scores[l], idx[l], count[l], out[l] if a_ else None, wss[wi], s_)

        def begin(l, s_, wi):
            hill.hill_evict_step_begin(desc, q_all[t][l], Kall[l % lres], lens_all[t], w.max_k, mode, acc(l),
                                       scores[l], wss[wi], s_)

        def end(l, s_, wi):
            hill.hill_evict_step_end(desc, lens_all[t], k_all[t], w.max_k, mode, acc(l), scores[l], idx[l],
                                     count[l], wss[wi], stream=s_)

        def attn(l, s_, wi):
            hill.hill_gather_sparse_attn(desc, q_all[t][l], Kall[l % lres], Vall[l % lres], idx[l], count[l],
                                         w.max_k, out[l], wsa[wi], s_)

        issue_layers(frm, L, st, side, att, with_attn, fused, begin, end, attn)

    tokens = sum(L * sum(w.lens_at(t)) for t in order)
    peak, _ = measured_peaks()
    piped = pipelined_form(mode, w.accumulate, lres)
    runs = [(piped, False), ("serial", False)] + ([(piped, True)] if full_step else [])
    res = {}
    for frm, with_attn in dict.fromkeys(runs):
        with torch.cuda.stream(stream):
            issue(steps_used[0], stream, frm, with_attn)
        hill.hill_sync_status(stream)
        graphs = [None] * S
        for t in steps_used:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                issue(t, stream, frm, with_attn)
            graphs[t] = g
        if accum is not None:
            accum.zero_()
        ms, clock_info = time_replays(graphs, order, args.warmup, stream, dev, clocks_of=local)
        ms = max_over_ranks(ms, dev)
        hill.hill_sync_status(stream)
        del graphs
        if with_attn:
            res["step"] = {"schedule": SCHEDULES[frm], "us_per_layer": round(ms * 1e3 / (len(order) * L), 2),
                           "tokens_per_s": round(world * tokens / (ms / 1e3), 1), "clocks": clock_info}
        else:
            res[frm] = dict(eval_summary(ms, tokens, Hkv * d * 2, len(order) * L, world, peak, frm), clocks=clock_info)
    # the scoring stage alone, per launch, at the last timed decode step
    t_s = order[-1]
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(L)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(L)]
    with torch.cuda.stream(stream):
        for rep in range(2):
            for l in range(L):
                if rep == 1:
                    starts[l].record(stream)
                hill.hill_score(desc, q_all[t_s][l], Kall[l % lres], lens_all[t_s], mode, scores[l], None, wss[0],
                                stream)
                if rep == 1:
                    ends[l].record(stream)
    stream.synchronize()
    hill.hill_sync_status(stream)
    score_us = sum(a.elapsed_time(b) for a, b in zip(starts, ends)) / L * 1e3
    out_d = dict(res[piped])
    if piped != "serial":
        out_d["serial"] = res["serial"]
    if full_step:
        out_d["step"] = res["step"]
    out_d.update({
        "workload": w.name, "batch": B, "heads": Hq, "kv_heads": Hkv, "kv_dtype": str(w.dtype).replace("torch.", ""),
        "tokens_last_step": w.lens_at(S - 1), "budget": f"floor({w.budget_frac}*len)" if w.budget_tokens is None
        else w.budget_tokens, "accumulate": w.accumulate, "layers": L, "layers_resident": lres,
        "decode_steps": S, "steps_timed": len(order),
        "scoring_stage_us": round(score_us, 2),
        "scoring_stage_frac_of_measured_hbm": round(
            sum(w.lens_at(t_s)) * (Hkv * d * 2 + 4) / (score_us / 1e6) / 1e9 / peak, 4),
        "generate_s": round(t_gen, 1),
    })
    del Kall, Vall, q_all, accum, scores, idx, count, out, wss, wsa
    torch.cuda.empty_cache()
    return out_d


def eval_select_only(args, n, hill, dev, world, mode):
    """The acceptance measurement of workload n (the contexts of 32K tokens
    or more the headline workload does not cover)."""
    rank, _, _ = dist_env()
    w, _ = workload_for(n, replica_seed(args.seed, rank), None)
    return measure_workload(args, w, hill, dev, world, mode)


def run_sweep(args):
    """The budget/batch sweep: B in {1, 8, 16} x {8K, 64K} tokens x budget in
    {5, 10, 20, 50} %, 32 layers, cumulative importance across decode steps;
    one JSON line per point (rank 0), resident layers reused cyclically where
    the point's KV does not fit in HBM."""
    import torch.distributed as dist

    from paper_2602_18750_gb300 import build as hbuild
    from paper_2602_18750_gb300 import hill

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    hbuild.build()
    hill.load()
    mode = hill.HILL_SCORE_ATTN if args.mode == "attn" else hill.HILL_SCORE_RAW
    for B in inputs.SWEEP_BATCHES:
        for n in inputs.SWEEP_LENS:
            for frac in inputs.SWEEP_BUDGETS:
                w = inputs.sweep_point(B, n, frac, seed=replica_seed(args.seed, rank))
                r = measure_workload(args, w, hill, dev, world, mode, full_step=True,
                                     layers_resident=args.layers_resident)
                if rank == 0:
                    print(json.dumps({"sweep_point": {"batch": B, "tokens": n, "budget_frac": frac},
                                      "metric": METRIC, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                                      "warmup": args.warmup, "importance": args.mode, **r}), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_e2e(args, w, lres, hill, desc, mode, Kall, Vall, q_all, lens_all, k_all, accum, scores, idx, count,
            out, wss, wsa, stream, dev, world, side, att, form):
    """Same steps through the public calls, in the bench's schedule (one
    fused hill_evict_step per layer, or the layer-pipelined begin / end plus
    hill_gather_sparse_attn on a second stream), with each step's inputs
    copied from pinned host memory (query of every layer, the new token's K/V
    row of every layer, lengths, budgets) and its results (selection and
    attention output of every layer) copied back, all inside the timed region."""
    L, S, B = w.layers, w.steps, w.batch
    order = [(args.warmup + i) % S for i in range(args.steps)]
    # host copies of what a caller would hold at each step
    q_h = torch.empty_like(q_all, device="cpu").pin_memory()
    q_h.copy_(q_all)
    pos = [[n - 1 for n in w.lens_at(t)] for t in range(S)]
    newk_h = torch.empty(S, lres, B, w.kv_heads, w.head_dim, dtype=w.dtype).pin_memory()
    newv_h = torch.empty_like(newk_h).pin_memory()
    for t in range(S):
        for b in range(B):
            newk_h[t, :, b].copy_(Kall[:, b, :, pos[t][b]])
            newv_h[t, :, b].copy_(Vall[:, b, :, pos[t][b]])
    lk_h = torch.stack([lens_all.cpu(), k_all.cpu()], 1).pin_memory()        # [S][2][B]
    lk_d = torch.empty(2, B, dtype=torch.int32, device=dev)
    stage_k = torch.empty(lres, B, w.kv_heads, w.head_dim, dtype=w.dtype, device=dev)
    stage_v = torch.empty_like(stage_k)
    idx_h = torch.empty_like(idx, device="cpu").pin_memory()
    cnt_h = torch.empty_like(count, device="cpu").pin_memory()
    out_h = torch.empty_like(out, device="cpu").pin_memory()
    pos_d = [torch.tensor(p, dtype=torch.long, device=dev) for p in pos]
    b_d = torch.arange(B, device=dev)
    # per-layer views, made once (as an engine would hold them)
    qv = [[q_all[t, l] for l in range(L)] for t in range(S)]
    Kv, Vv = [Kall[r] for r in range(lres)], [Vall[r] for r in range(lres)]
    accv = [accum[r] if accum is not None else None for r in range(lres)]
    scv = list(scores)

    def compute(t, lens_d, kk_d, ri, rc, ro):
        """The step's calls on the device buffers: lengths/budgets lens_d,
        kk_d; results into the per-layer views ri, rc, ro."""
        def fused(l, with_attn, st, wi):
            r = l % lres
            hill.hill_evict_step(desc, qv[t][l], Kv[r], Vv[r], lens_d, kk_d, w.max_k, mode, accv[r], scv[l], ri[l],
                                 rc[l], ro[l] if with_attn else None, wss[wi], st)

        def begin(l, st, wi):
            hill.hill_evict_step_begin(desc, qv[t][l], Kv[l % lres], lens_d, w.max_k, mode, accv[l % lres], scv[l],
                                       wss[wi], st)

        def end(l, st, wi):
            hill.hill_evict_step_end(desc, lens_d, kk_d, w.max_k, mode, accv[l % lres], scv[l], ri[l], rc[l],
                                     wss[wi], stream=st)

        def attn(l, st, wi):
            r = l % lres
            hill.hill_gather_sparse_attn(desc, qv[t][l], Kv[r], Vv[r], ri[l], rc[l], w.max_k, ro[l], wsa[wi], st)

        issue_layers(form, L, stream, side, att, True, fused, begin, end, attn)

    def append(t, sk, sv):
        # the new token's K/V row of every resident layer and sequence, one
        # indexed write per cache: K[:, b, :, pos[b]] = sk[:, b] for every b
        Kall[:, b_d, :, pos_d[t]] = sk.transpose(0, 1)
        Vall[:, b_d, :, pos_d[t]] = sv.transpose(0, 1)

    res0 = (list(idx), list(count), list(out))

    def one(t):
        q_all[t].copy_(q_h[t], non_blocking=True)
        stage_k.copy_(newk_h[t], non_blocking=True)
        stage_v.copy_(newv_h[t], non_blocking=True)
        lk_d.copy_(lk_h[t], non_blocking=True)
        append(t, stage_k, stage_v)
        compute(t, lk_d[0], lk_d[1], *res0)
        idx_h.copy_(idx, non_blocking=True)
        cnt_h.copy_(count, non_blocking=True)
        out_h.copy_(out, non_blocking=True)

    # Overlapped form (what a serving loop does): while step t computes, a copy
    # stream brings in step t + 1's inputs -- its queries, lengths and budgets,
    # and its new K/V rows, written into the caches at once -- and copies out
    # step t - 1's results.  Inputs are staged and results written in two
    # alternating buffer sets, so a step's compute never touches the buffers
    # being copied; the new rows of step t + 1 lie at or past step t's
    # lengths, where step t's kernels use no key or value.
    cstream = torch.cuda.Stream(device=dev)
    stage2_k = torch.empty((2,) + tuple(stage_k.shape), dtype=w.dtype, device=dev)
    stage2_v = torch.empty_like(stage2_k)
    lk2_d = torch.empty(2, 2, B, dtype=torch.int32, device=dev)
    res = [(idx, count, out), (torch.empty_like(idx), torch.empty_like(count), torch.empty_like(out))]
    resv = [(list(a), list(c), list(o)) for a, c, o in res]
    cfork, cjoin = torch.cuda.Event(), torch.cuda.Event()

    def stage_in(t, par):
        q_all[t].copy_(q_h[t], non_blocking=True)
        stage2_k[par].copy_(newk_h[t], non_blocking=True)
        stage2_v[par].copy_(newv_h[t], non_blocking=True)
        lk2_d[par].copy_(lk_h[t], non_blocking=True)

    def one_overlapped(t, par):
        cfork.record(stream)
        cstream.wait_event(cfork)
        with torch.cuda.stream(cstream):
            stage_in((t + 1) % S, 1 - par)
            append((t + 1) % S, stage2_k[1 - par], stage2_v[1 - par])
            pi, pc, po = res[1 - par]
            idx_h.copy_(pi, non_blocking=True)
            cnt_h.copy_(pc, non_blocking=True)
            out_h.copy_(po, non_blocking=True)
        cjoin.record(cstream)
        compute(t, lk2_d[par][0], lk2_d[par][1], *resv[par])
        stream.wait_event(cjoin)

    def timed(step_fn):
        """step_fn(i) runs the i-th executed step (decode step i % S); the
        warm-up steps come first, then exactly the timed ones (`order`)."""
        with torch.cuda.stream(stream):
            for i in range(args.warmup):
                step_fn(i)
        stream.synchronize()
        barrier(dev)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for i in range(args.warmup, args.warmup + len(order)):
                step_fn(i)
            e1.record(stream)
        stream.synchronize()
        barrier(dev)
        hill.hill_sync_status(stream)
        return max_over_ranks(e0.elapsed_time(e1), dev)

    # eager: every copy and call issued from Python at every step, in order
    ms_eager = timed(lambda i: one(i % S))
    # captured once per decode step (and buffer parity) and replayed, the
    # copies overlapped with the compute as above
    with torch.cuda.stream(stream):
        stage_in(0, 0)
        append(0, stage2_k[0], stage2_v[0])
    stream.synchronize()
    graphs = {}
    for i in range(args.warmup + len(order)):
        key = (i % S, i % 2)
        if key not in graphs and S > 1:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                one_overlapped(*key)
            graphs[key] = g
    if S > 1:
        ms = timed(lambda i: graphs[(i % S, i % 2)].replay())
    else:
        # a single decode step cannot stage its successor: copies in line
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            one(0)
        graphs[(0, 0)] = g
        ms = timed(lambda i: g.replay())
    del graphs
    tokens = sum(L * sum(w.lens_at(t)) for t in order)
    h2d = (q_h[0].numel() * q_h.element_size() + 2 * newk_h[0].numel() * newk_h.element_size()
           + lk_h[0].numel() * 4)
    d2h = idx_h.numel() * 4 + cnt_h.numel() * 4 + out_h.numel() * 4
    calls = SCHEDULES[form]
    return {"value": round(world * tokens / (ms / 1e3), 1), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": round(ms / len(order), 4),
            "api": calls + "; captured per decode step in a CUDA graph and replayed; every step copies one "
                           "step's inputs in from pinned host memory (writing its new K/V rows into the caches) "
                           "and one step's results out to pinned host memory on a copy stream, overlapped with "
                           "the compute (next step's inputs, previous step's results; two alternating buffer "
                           "sets)",
            "eager": {"value": round(world * tokens / (ms_eager / 1e3), 1),
                      "ms_per_step": round(ms_eager / len(order), 4),
                      "api": calls + "; issued from Python at every step (no graph)"}}


def cpu_baseline(w, lres, Kall, Vall, q_all, mode, seconds=10.0):
    """The oracle as it stands on the host cores, on (layer, step) samples of
    the same workload until about `seconds` of CPU time have run."""
    import oracle
    oracle.build()
    done_tokens, spent, samples = 0, 0.0, []
    for i in range(w.layers * w.steps):
        l, t = i % w.layers, (i * 7) % w.steps
        r = l % lres
        lens, k = w.lens_at(t), w.budget_at(t)
        q = q_all[t, l].cpu()
        K, V = Kall[r].cpu(), Vall[r].cpu()
        t0 = time.perf_counter()
        oracle.evict_step(mode, q, K, V, lens, k, w.max_k, with_attn=True)
        spent += time.perf_counter() - t0
        done_tokens += sum(lens)
        samples.append(f"L{l}/t{t}")
        if spent >= seconds:
            break
    return {"value": round(done_tokens / spent, 1), "unit": UNIT, "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"{len(samples)} (layer, decode step) evaluations of the same workload "
                      f"({', '.join(samples[:4])}{', ...' if len(samples) > 4 else ''}), all {w.batch} "
                      f"sequences, score + top-k + sparse attention in float64, {spent:.1f} s"}


# ---------------------------------------------------------------- reference arm (the oracle)
def run_reference(args):
    """The oracle on the host cores, as it stands: each step is one (layer,
    decode step) evaluation of the workload (all sequences)."""
    import oracle
    rank, world, _ = dist_env()
    if rank != 0:
        return
    oracle.build()
    w, lres = workload_for(args.workload, args.seed, args.layers_resident, args.kv_heads)
    lres = min(lres, 2)   # a couple of distinct layers, generated on the host
    caches = [inputs.layer_cache(w, l, device="cpu") for l in range(lres)]
    mode = oracle.ATTN if args.mode == "attn" else oracle.RAW

    def step(i):
        l, t = i % w.layers, i % w.steps
        K, V = caches[l % lres]
        q = inputs.step_query(w, l, t, device="cpu")
        lens, k = w.lens_at(t), w.budget_at(t)
        oracle.evict_step(mode, q, K, V, lens, k, w.max_k, with_attn=True)
        return sum(lens)

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    tokens = 0
    for i in range(args.steps):
        tokens += step(args.warmup + i)
    sec = time.perf_counter() - t0
    value = tokens / sec
    cores = oracle.num_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(sec * 1e3 / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": describe(w, lres, args.mode),
        "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "each step: one (layer, decode step) of the workload, all "
                                   f"{w.batch} sequences, score + top-k + sparse attention"},
        "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", type=int, default=3,
                    help="1..5 (default 3: B 4 x 16-32K ragged, the Qwen-7B stack)")
    ap.add_argument("--mode", choices=["attn", "raw"], default="attn")
    ap.add_argument("--kv-heads", type=int, default=None,
                    help="another head layout of the workload: its query heads over this many KV heads "
                         "(e.g. 1 for MQA)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--layers-resident", type=int, default=None,
                    help="allocate this many layers and cycle them (workloads larger than HBM)")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="the budget/batch sweep (B x tokens x budget, accumulating): one JSON line per point")
    ap.add_argument("--no-acceptance", action="store_true",
                    help="skip timing evaluation + selection on the other 32K+ workloads")
    ap.add_argument("--serial", action="store_true",
                    help="time the serial schedule (one fused hill_evict_step per layer) as the headline; the "
                         "default is the layer-pipelined schedule of Sec. 4.3 (both are measured and reported)")
    ap.add_argument("--f8", action="store_true",
                    help="asymmetric-precision scoring (Sec. 4.4) from an E4M3 key shadow (hill_evict_step_f8)")
    ap.add_argument("--bkp-recent", type=int, default=-1,
                    help="BKP bookkeeping (Sec. 4.2): pin this many recent tokens and keep a hit-rate table "
                         "(hill_evict_step_bkp); default off")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()

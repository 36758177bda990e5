"""Thin ctypes binding over libhill's C ABI (include/hill.h).

Every function here only marshals arguments: tensors become device pointers,
a descriptor is filled from tensor shapes and strides, and a non-OK status
raises :class:`HillError`.  All arithmetic runs in the CUDA kernels of
libhill.so; there is no other implementation behind these names, and loading
fails loudly if the library has not been built.

Names follow the C ABI: :func:`hill_score`, :func:`hill_topk_select`,
:func:`hill_gather_sparse_attn`, :func:`hill_evict_step`, :func:`hill_topk_select_bkp`,
:func:`hill_evict_step_bkp`, :func:`hill_quantize_k`, :func:`hill_score_f8`, :func:`hill_evict_step_f8`,
:func:`hill_evict_step_kvh`, :func:`hill_evict_step_begin`, :func:`hill_evict_step_begin_f8`,
:func:`hill_evict_step_end`, :func:`hill_workspace_bytes`, :func:`hill_sync_status`.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

HILL_OK = 0
HILL_ERR_INVALID_ARG = 1
HILL_ERR_UNSUPPORTED = 2
HILL_ERR_WORKSPACE = 3
HILL_ERR_CUDA = 4
HILL_ERR_TIMEOUT = 5
HILL_ERR_DEVICE = 6

HILL_F16, HILL_BF16 = 0, 1
HILL_SCORE_ATTN, HILL_SCORE_RAW = 0, 1

LIB_PATH = _build.LIB


class HillError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


class hill_desc(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("capacity", ctypes.c_int32), ("dtype", ctypes.c_int32),
        ("q_sb", ctypes.c_int64), ("q_sh", ctypes.c_int64),
        ("k_sb", ctypes.c_int64), ("k_sh", ctypes.c_int64), ("k_sn", ctypes.c_int64),
        ("v_sb", ctypes.c_int64), ("v_sh", ctypes.c_int64), ("v_sn", ctypes.c_int64),
    ]


_lib = None


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libhill.so (raises OSError if it is missing: build it first)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise OSError(f"libhill.so not built ({path}); run python -m paper_2602_18750_gb300.build")
    lib = ctypes.CDLL(path)
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    D = ctypes.POINTER(hill_desc)
    lib.hill_workspace_bytes.argtypes = [D, I32, I32]
    lib.hill_workspace_bytes.restype = SZ
    lib.hill_score.argtypes = [D, P, P, P, I32, P, P, P, SZ, P]
    lib.hill_topk_select.argtypes = [D, P, P, P, I32, P, P, P, SZ, P]
    lib.hill_gather_sparse_attn.argtypes = [D, P, P, P, P, P, I32, P, P, SZ, P]
    lib.hill_evict_step.argtypes = [D, P, P, P, P, P, I32, I32, P, P, P, P, P, P, SZ, P]
    lib.hill_topk_select_bkp.argtypes = [D, P, P, P, I32, I32, P, P, P, P, SZ, P]
    lib.hill_evict_step_bkp.argtypes = [D, P, P, P, P, P, I32, I32, I32, P, P, P, P, P, P, P, SZ, P]
    lib.hill_quantize_k.argtypes = [D, P, P, P, I32, P, P, P]
    lib.hill_evict_step_kvh.argtypes = [D, P, P, P, P, P, I32, I32, P, P, P, P, P, P, SZ, P]
    lib.hill_evict_step_begin.argtypes = [D, P, P, P, I32, I32, P, P, P, SZ, P]
    lib.hill_evict_step_begin_f8.argtypes = [D, P, P, P, P, I32, I32, P, P, P, SZ, P]
    lib.hill_evict_step_end.argtypes = [D, P, P, I32, I32, I32, P, P, P, P, P, P, SZ, P]
    lib.hill_selftest_wait.argtypes = [ctypes.c_uint32, P]
    lib.hill_score_f8.argtypes = [D, P, P, P, P, I32, P, P, P, SZ, P]
    lib.hill_evict_step_f8.argtypes = [D, P, P, P, P, P, P, P, I32, I32, P, P, P, P, P, P, SZ, P]
    lib.hill_score_noalloc.argtypes = [D, P, P, P, I32, P, P, P]
    lib.hill_score_noalloc.restype = I32
    lib.hill_sync_status.argtypes = [P]
    lib.hill_status_string.argtypes = [I32]
    lib.hill_status_string.restype = ctypes.c_char_p
    lib.hill_abi_version.restype = I32
    lib.hill_kernel_launches.restype = ctypes.c_uint64
    for name in ("hill_score", "hill_topk_select", "hill_gather_sparse_attn", "hill_evict_step",
                 "hill_topk_select_bkp", "hill_evict_step_bkp", "hill_quantize_k", "hill_score_f8",
                 "hill_evict_step_f8", "hill_evict_step_kvh", "hill_evict_step_begin", "hill_evict_step_begin_f8",
                 "hill_evict_step_end", "hill_selftest_wait", "hill_sync_status"):
        getattr(lib, name).restype = I32
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().hill_status_string(int(status)).decode()


def _check(status: int, where: str) -> None:
    if status != HILL_OK:
        raise HillError(status, where)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_desc(q: torch.Tensor, k_cache: torch.Tensor, v_cache: torch.Tensor | None = None) -> hill_desc:
    """Descriptor from q [B][H][d] and K/V [B][Hkv][cap][d] (any element strides, d contiguous)."""
    B, H, d = q.shape
    Bk, Hkv, cap, dk = k_cache.shape
    if Bk != B or dk != d:
        raise ValueError(f"shape mismatch q {tuple(q.shape)} vs K {tuple(k_cache.shape)}")
    if q.stride(-1) != 1 or k_cache.stride(-1) != 1:
        raise ValueError("head dimension must be contiguous")
    if q.dtype != k_cache.dtype:
        raise ValueError("q and K must share a dtype")
    dt = {torch.float16: HILL_F16, torch.bfloat16: HILL_BF16}.get(q.dtype)
    if dt is None:
        raise ValueError(f"unsupported dtype {q.dtype}")
    v = v_cache if v_cache is not None else k_cache
    if tuple(v.shape) != tuple(k_cache.shape) or v.stride(-1) != 1 or v.dtype != q.dtype:
        raise ValueError("V must match K in shape and dtype")
    return hill_desc(B, H, Hkv, d, cap, dt,
                     q.stride(0), q.stride(1),
                     k_cache.stride(0), k_cache.stride(1), k_cache.stride(2),
                     v.stride(0), v.stride(1), v.stride(2))


def hill_workspace_bytes(desc: hill_desc, mode: int, max_k: int) -> int:
    return int(load().hill_workspace_bytes(ctypes.byref(desc), int(mode), int(max_k)))


def alloc_workspace(desc: hill_desc, mode: int, max_k: int, device="cuda") -> torch.Tensor:
    n = hill_workspace_bytes(desc, mode, max_k)
    if n == 0:
        raise HillError(HILL_ERR_INVALID_ARG, "hill_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def _ws(ws):
    if ws is None:
        return None, 0
    return ws.data_ptr(), ws.numel() * ws.element_size()


def hill_score(desc, q, k_cache, lens, mode, scores, accum=None, ws=None, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_score(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(lens), int(mode),
                             _ptr(scores), _ptr(accum), wp, wn, _stream(stream)), "hill_score")


def hill_score_noalloc(desc, q, k_cache, lens, mode, scores, accum=None, stream=None) -> None:
    """hill_score without a workspace: scratch lives in a fixed array inside
    the library (for callers that cannot allocate device memory)."""
    _check(load().hill_score_noalloc(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(lens), int(mode),
                                     _ptr(scores), _ptr(accum), _stream(stream)), "hill_score_noalloc")


def hill_topk_select(desc, scores, lens, k, max_k, idx, count, ws=None, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_topk_select(ctypes.byref(desc), _ptr(scores), _ptr(lens), _ptr(k), int(max_k),
                                   _ptr(idx), _ptr(count), wp, wn, _stream(stream)), "hill_topk_select")


def hill_gather_sparse_attn(desc, q, k_cache, v_cache, idx, count, max_k, out, ws=None, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_gather_sparse_attn(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(v_cache),
                                          _ptr(idx), _ptr(count), int(max_k), _ptr(out), wp, wn,
                                          _stream(stream)), "hill_gather_sparse_attn")


def hill_evict_step(desc, q, k_cache, v_cache, lens, k, max_k, mode, accum, scores, idx, count, out,
                    ws, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_evict_step(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(lens),
                                  _ptr(k), int(max_k), int(mode), _ptr(accum), _ptr(scores), _ptr(idx),
                                  _ptr(count), _ptr(out), wp, wn, _stream(stream)), "hill_evict_step")


def hill_topk_select_bkp(desc, scores, lens, k, recent, max_k, idx, count, hits=None, ws=None,
                         stream=None) -> None:
    """BKP selection (Sec. 4.2): the `recent` newest tokens pinned, the top-k of
    the older ones, and hits[b][j] += 1 (saturating uint16) for kept tokens."""
    wp, wn = _ws(ws)
    _check(load().hill_topk_select_bkp(ctypes.byref(desc), _ptr(scores), _ptr(lens), _ptr(k), int(recent),
                                       int(max_k), _ptr(idx), _ptr(count), _ptr(hits), wp, wn,
                                       _stream(stream)), "hill_topk_select_bkp")


def hill_evict_step_bkp(desc, q, k_cache, v_cache, lens, k, recent, max_k, mode, accum, scores, idx, count,
                        hits, out, ws, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_bkp(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(lens),
                                      _ptr(k), int(recent), int(max_k), int(mode), _ptr(accum), _ptr(scores),
                                      _ptr(idx), _ptr(count), _ptr(hits), _ptr(out), wp, wn,
                                      _stream(stream)), "hill_evict_step_bkp")


def hill_evict_step_begin(desc, q, k_cache, lens, max_k, mode, accum, scores, ws, stream=None) -> None:
    """First half of the split step: the scoring kernel (K stream)."""
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_begin(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(lens), int(max_k),
                                        int(mode), _ptr(accum), _ptr(scores), wp, wn, _stream(stream)),
           "hill_evict_step_begin")


def hill_evict_step_begin_f8(desc, q, k8, kscale, lens, max_k, mode, accum, scores, ws, stream=None) -> None:
    """First half of the split step from the E4M3 key shadow."""
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_begin_f8(ctypes.byref(desc), _ptr(q), _ptr(k8), _ptr(kscale), _ptr(lens),
                                           int(max_k), int(mode), _ptr(accum), _ptr(scores), wp, wn,
                                           _stream(stream)), "hill_evict_step_begin_f8")


def hill_evict_step_end(desc, lens, k, max_k, mode, accum, scores, idx, count, ws, recent=0, hits=None,
                        stream=None) -> None:
    """Second half of the split step: normalisation (ATTN) and selection."""
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_end(ctypes.byref(desc), _ptr(lens), _ptr(k), int(recent), int(max_k), int(mode),
                                      _ptr(accum), _ptr(scores), _ptr(idx), _ptr(count), _ptr(hits), wp, wn,
                                      _stream(stream)), "hill_evict_step_end")


def hill_evict_step_kvh(desc, q, k_cache, v_cache, lens, k, max_k, mode, accum, scores, idx, count, out, ws,
                        stream=None) -> None:
    """Per-KV-head selection: scores [B][Hkv][cap], idx [B][Hkv][max_k], count [B][Hkv]."""
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_kvh(ctypes.byref(desc), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(lens),
                                      _ptr(k), int(max_k), int(mode), _ptr(accum), _ptr(scores), _ptr(idx),
                                      _ptr(count), _ptr(out), wp, wn, _stream(stream)), "hill_evict_step_kvh")


def shadow_shape(desc):
    """Shapes of the E4M3 key shadow: (codes [B][Hkv][cap][128], scales [B][Hkv][cap32])."""
    cap32 = (desc.capacity + 31) // 32 * 32
    return ((desc.batch, desc.num_kv_heads, desc.capacity, desc.head_dim),
            (desc.batch, desc.num_kv_heads, cap32))


def alloc_shadow(desc, device="cuda"):
    cs, ss = shadow_shape(desc)
    return torch.zeros(cs, dtype=torch.uint8, device=device), torch.zeros(ss, dtype=torch.float32, device=device)


def hill_quantize_k(desc, k_cache, row_begin, row_end, max_rows, k8, kscale, stream=None) -> None:
    _check(load().hill_quantize_k(ctypes.byref(desc), _ptr(k_cache), _ptr(row_begin), _ptr(row_end),
                                  int(max_rows), _ptr(k8), _ptr(kscale), _stream(stream)), "hill_quantize_k")


def hill_score_f8(desc, q, k8, kscale, lens, mode, scores, accum=None, ws=None, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_score_f8(ctypes.byref(desc), _ptr(q), _ptr(k8), _ptr(kscale), _ptr(lens), int(mode),
                                _ptr(scores), _ptr(accum), wp, wn, _stream(stream)), "hill_score_f8")


def hill_evict_step_f8(desc, q, k8, kscale, k_cache, v_cache, lens, k, max_k, mode, accum, scores, idx, count,
                       out, ws, stream=None) -> None:
    wp, wn = _ws(ws)
    _check(load().hill_evict_step_f8(ctypes.byref(desc), _ptr(q), _ptr(k8), _ptr(kscale), _ptr(k_cache),
                                     _ptr(v_cache), _ptr(lens), _ptr(k), int(max_k), int(mode), _ptr(accum),
                                     _ptr(scores), _ptr(idx), _ptr(count), _ptr(out), wp, wn, _stream(stream)),
           "hill_evict_step_f8")


def hill_selftest_wait(limit_us: int, stream=None) -> None:
    """Run the bounded-wait self test (its expiry shows up in hill_sync_status)."""
    _check(load().hill_selftest_wait(int(limit_us), _stream(stream)), "hill_selftest_wait")


def hill_kernel_launches() -> int:
    return int(load().hill_kernel_launches())


def hill_sync_status(stream=None) -> None:
    _check(load().hill_sync_status(_stream(stream)), "hill_sync_status")


class Evictor:
    """Holds the workspace and output buffers for repeated steps of one shape.

    ``step()`` issues exactly one hill_evict_step call; buffers are allocated
    once with torch (device memory plumbing only).
    """

    def __init__(self, q, k_cache, v_cache, max_k: int, mode: int = HILL_SCORE_ATTN,
                 with_scores: bool = True, with_attn: bool = True):
        self.desc = make_desc(q, k_cache, v_cache)
        self.mode = int(mode)
        self.max_k = int(max_k)
        dev = q.device
        B, H, d = q.shape
        cap = k_cache.shape[2]
        self.ws = alloc_workspace(self.desc, self.mode, self.max_k, dev)
        self.scores = torch.empty(B, cap, dtype=torch.float32, device=dev) if with_scores else None
        self.idx = torch.empty(B, max(self.max_k, 1), dtype=torch.int32, device=dev)
        self.count = torch.empty(B, dtype=torch.int32, device=dev)
        self.out = torch.empty(B, H, d, dtype=torch.float32, device=dev) if with_attn else None

    def step(self, q, k_cache, v_cache, lens, k, accum=None, stream=None):
        hill_evict_step(self.desc, q, k_cache, v_cache, lens, k, self.max_k, self.mode, accum,
                        self.scores, self.idx, self.count, self.out, self.ws, stream)
        return self

"""CPU oracle for HillInfer's token-importance evaluation (arxiv 2602.18750).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` are the only
callers.  The product path (the CUDA library and its binding) never imports
this package, and this package imports nothing from the product.

The arithmetic lives in ``hill_oracle.c`` (plain C, float64 on the exact
16-bit input values); this module only compiles it with gcc and marshals numpy
arrays into it.  Each wrapper names the part of the paper it follows:

* :func:`logits`       -- Eq. 1 (Sec. 2.1), q.K^T / sqrt(d) over the whole cache
* :func:`logits_q8`    -- the same from E4M3 operands (Sec. 4.4 asymmetric precision),
                          with :func:`quantize_rows`, :func:`e4m3_encode`, :func:`e4m3_decode`
* :func:`scores`       -- Sec. 4.1 (column sum of softmax weights, ATTN) and
                          Sec. 4.4 (raw inner product, RAW)
* :func:`accumulate`   -- running importance across decode steps (Sec. 4.2)
* :func:`topk`         -- top-alpha selection (Sec. 3.1, Sec. 4.2)
* :func:`bkp_select`   -- BKP pinning + hit-rate table (Sec. 4.2)
* :func:`sparse_attn`  -- attention over the selected KV only (Sec. 4.1, workflow step 6)
* :func:`evict_step`   -- the five steps in order
* :func:`scores_kvh`, :func:`topk_kvh`, :func:`sparse_attn_kvh` -- the per-KV-head
                          selection variant, composed from the functions above

Pins: tests/test_oracle_pins.py checks every function against library
routines (torch fp64 matmul / softmax / topk / scaled_dot_product_attention),
closed forms, invariants and hand-derived golden cases.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hill_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")

F16, BF16 = 0, 1
ATTN, RAW = 0, 1

_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile hill_oracle.c into oracle/_build/liboracle.so with gcc.

    OpenMP is used when the compiler supports it (the (b, h) loops of the
    logits and the attention are independent); otherwise the build is serial.
    """
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            P = ctypes.c_void_p
            I = ctypes.c_int
            lib.oracle_logits.argtypes = [I, I, I, I, I, I, P, P, P, P]
            lib.oracle_scores.argtypes = [I, I, I, I, P, P, P]
            lib.oracle_accumulate.argtypes = [I, I, P, P, P]
            lib.oracle_topk.argtypes = [I, I, P, P, P, I, P, P]
            lib.oracle_bkp_select.argtypes = [I, I, P, P, P, I, I, P, P, P]
            lib.oracle_sparse_attn.argtypes = [I, I, I, I, I, I, P, P, P, P, P, I, P]
            lib.oracle_evict_step.argtypes = [I, I, I, I, I, I, I, P, P, P, P, P, I,
                                              P, P, P, P, P, P]
            lib.oracle_decode16_array.argtypes = [I, P, P, ctypes.c_int64]
            lib.oracle_e4m3_decode_array.argtypes = [P, P, ctypes.c_int64]
            lib.oracle_e4m3_decode_array.restype = None
            lib.oracle_e4m3_encode_array.argtypes = [P, P, ctypes.c_int64]
            lib.oracle_e4m3_encode_array.restype = None
            lib.oracle_quantize_rows.argtypes = [I, ctypes.c_int64, I, P, P, P]
            lib.oracle_quantize_rows.restype = None
            lib.oracle_logits_q8.argtypes = [I, I, I, I, I, I, P, P, P, P, P]
            lib.oracle_decode16_array.restype = None
            lib.oracle_accumulate.restype = None
            lib.oracle_num_threads.restype = I
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _bits(x) -> np.ndarray:
    """16-bit float tensor/array -> contiguous uint16 array of its bit patterns."""
    if isinstance(x, np.ndarray):
        if x.dtype == np.float16:
            return np.ascontiguousarray(x).view(np.uint16)
        if x.dtype == np.uint16:
            return np.ascontiguousarray(x)
        raise TypeError(f"unsupported array dtype {x.dtype}")
    import torch  # only for tensors handed in by the tests
    t = x.detach().to("cpu").contiguous()
    if t.dtype not in (torch.float16, torch.bfloat16):
        raise TypeError(f"unsupported tensor dtype {t.dtype}")
    return t.view(torch.int16).numpy().view(np.uint16)


def _dtype_code(x, dtype):
    if dtype is not None:
        return dtype
    if isinstance(x, np.ndarray):
        return F16
    import torch
    return BF16 if x.dtype == torch.bfloat16 else F16


def _i32(a) -> np.ndarray:
    if not isinstance(a, np.ndarray):
        a = np.asarray(a.detach().cpu() if hasattr(a, "detach") else a)
    return np.ascontiguousarray(a, dtype=np.int32)


def num_threads() -> int:
    return _load().oracle_num_threads()


def decode16(x, dtype=None) -> np.ndarray:
    """Exact float64 values of 16-bit inputs, decoded by the oracle's own decoder."""
    code = _dtype_code(x, dtype)
    bits = _bits(x)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_decode16_array(code, _ptr(bits), _ptr(out), bits.size)
    return out


def e4m3_decode(codes) -> np.ndarray:
    """Exact float64 values of E4M3 codes (uint8)."""
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    out = np.empty(c.shape, dtype=np.float64)
    _load().oracle_e4m3_decode_array(_ptr(c), _ptr(out), c.size)
    return out


def e4m3_encode(x) -> np.ndarray:
    """Nearest E4M3 codes of float32 values (ties to even, saturating at 448)."""
    v = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(v.shape, dtype=np.uint8)
    _load().oracle_e4m3_encode_array(_ptr(v), _ptr(out), v.size)
    return out


def quantize_rows(x, dtype=None):
    """Rows of the last dimension of a 16-bit tensor -> (codes uint8, scale float32)."""
    code = _dtype_code(x, dtype)
    bits = _bits(x)
    d = bits.shape[-1]
    rows = bits.size // d
    codes = np.empty(bits.shape, dtype=np.uint8)
    scale = np.empty(bits.shape[:-1], dtype=np.float32)
    _load().oracle_quantize_rows(code, rows, d, _ptr(bits), _ptr(codes), _ptr(scale))
    return codes, scale


def logits_q8(q, kcodes, kscale, lens, dtype=None) -> np.ndarray:
    """z8[B][H][cap] (NaN where j >= lens[b]) from the 8-bit operands (Sec. 4.4)."""
    code = _dtype_code(q, dtype)
    qb = _bits(q)
    kc = np.ascontiguousarray(kcodes, dtype=np.uint8)
    ks = np.ascontiguousarray(kscale, dtype=np.float32)
    B, H, d = qb.shape
    _, Hkv, cap, d2 = kc.shape
    assert d2 == d and ks.shape == (B, Hkv, cap)
    z = np.full((B, H, cap), np.nan)
    rc = _load().oracle_logits_q8(code, B, H, Hkv, d, cap, _ptr(qb), _ptr(kc), _ptr(ks), _ptr(_i32(lens)),
                                  _ptr(z))
    if rc:
        raise ValueError(f"oracle_logits_q8 rc={rc}")
    return z


def logits(q, K, lens, dtype=None) -> np.ndarray:
    """z[B][H][cap] (NaN where j >= lens[b]); q [B][H][d], K [B][Hkv][cap][d]."""
    code = _dtype_code(q, dtype)
    qb, kb = _bits(q), _bits(K)
    B, H, d = qb.shape
    _, Hkv, cap, d2 = kb.shape
    assert d2 == d and kb.shape[0] == B
    ln = _i32(lens)
    z = np.full((B, H, cap), np.nan)
    rc = _load().oracle_logits(code, B, H, Hkv, d, cap, _ptr(qb), _ptr(kb), _ptr(ln), _ptr(z))
    if rc:
        raise ValueError(f"oracle_logits rc={rc}")
    return z


def scores(mode, z, lens) -> np.ndarray:
    """s[B][cap] (NaN where j >= lens[b]) from logits z[B][H][cap]."""
    z = np.ascontiguousarray(z, dtype=np.float64)
    B, H, cap = z.shape
    ln = _i32(lens)
    s = np.full((B, cap), np.nan)
    rc = _load().oracle_scores(mode, B, H, cap, _ptr(ln), _ptr(z), _ptr(s))
    if rc:
        raise ValueError(f"oracle_scores rc={rc}")
    return s


def accumulate(s, A, lens) -> np.ndarray:
    """Return A + s on j < lens[b] (A unchanged elsewhere); A is not modified."""
    s = np.ascontiguousarray(s, dtype=np.float64)
    out = np.array(A, dtype=np.float64, copy=True, order="C")
    B, cap = s.shape
    _load().oracle_accumulate(B, cap, _ptr(_i32(lens)), _ptr(s), _ptr(out))
    return out


def topk(key, lens, k, max_k):
    """(idx[B][max_k], count[B], rc); key [B][cap] (float32 keys are exact in float64)."""
    key = np.ascontiguousarray(key, dtype=np.float64)
    B, cap = key.shape
    idx = np.full((B, max_k), -7, dtype=np.int32)
    count = np.zeros(B, dtype=np.int32)
    rc = _load().oracle_topk(B, cap, _ptr(_i32(lens)), _ptr(key), _ptr(_i32(k)), max_k,
                             _ptr(idx), _ptr(count))
    return idx, count, rc


def bkp_select(key, lens, k, recent, max_k, hits=None):
    """BKP selection (Sec. 4.2): pinned recent window + top-k of the older
    tokens.  Returns (idx[B][max_k], count[B], rc, hits') with hits' a
    uint16 copy of `hits` after the step's increments (None if hits is None)."""
    key = np.ascontiguousarray(key, dtype=np.float64)
    B, cap = key.shape
    idx = np.full((B, max_k), -7, dtype=np.int32)
    count = np.zeros(B, dtype=np.int32)
    h = None if hits is None else np.array(hits, dtype=np.uint16, copy=True, order="C")
    rc = _load().oracle_bkp_select(B, cap, _ptr(_i32(lens)), _ptr(key), _ptr(_i32(k)), int(recent),
                                   max_k, _ptr(idx), _ptr(count), _ptr(h))
    return idx, count, rc, h


def scores_kvh(mode, z, lens, Hkv) -> np.ndarray:
    """Per-KV-head importance s[B][Hkv][cap]: Step 2 restricted to the G query
    heads of each KV head (the same softmax per (b, h), summed within the
    group only), i.e. :func:`scores` on z regrouped as [B*Hkv][G][cap]."""
    z = np.ascontiguousarray(z, dtype=np.float64)
    B, H, cap = z.shape
    G = H // Hkv
    s = scores(mode, z.reshape(B * Hkv, G, cap), np.repeat(_i32(lens), Hkv))
    return s.reshape(B, Hkv, cap)


def topk_kvh(key, lens, k, max_k):
    """One top-k per (b, g) row of key[B][Hkv][cap] (budget k[b] for every g):
    (idx[B][Hkv][max_k], count[B][Hkv], rc)."""
    key = np.ascontiguousarray(key, dtype=np.float64)
    B, Hkv, cap = key.shape
    idx, count, rc = topk(key.reshape(B * Hkv, cap), np.repeat(_i32(lens), Hkv), np.repeat(_i32(k), Hkv), max_k)
    return idx.reshape(B, Hkv, max_k), count.reshape(B, Hkv), rc


def sparse_attn_kvh(q, K, V, idx, count, dtype=None) -> np.ndarray:
    """Attention where the query heads of KV head g read only the rows
    idx[b][g][:count[b][g]]: :func:`sparse_attn` per KV head."""
    Hkv = K.shape[1]
    H = q.shape[1]
    G = H // Hkv
    idx = np.asarray(idx)
    count = np.asarray(count)
    outs = [sparse_attn(q[:, g * G:(g + 1) * G], K[:, g:g + 1], V[:, g:g + 1], idx[:, g], count[:, g], dtype)
            for g in range(Hkv)]
    return np.concatenate(outs, axis=1)


def sparse_attn(q, K, V, idx, count, dtype=None) -> np.ndarray:
    """out[B][H][d] float64: softmax attention of q over the rows idx[b][:count[b]]."""
    code = _dtype_code(q, dtype)
    qb, kb, vb = _bits(q), _bits(K), _bits(V)
    B, H, d = qb.shape
    _, Hkv, cap, _ = kb.shape
    idx = _i32(idx)
    max_k = idx.shape[1] if idx.ndim == 2 else 0
    out = np.zeros((B, H, d))
    rc = _load().oracle_sparse_attn(code, B, H, Hkv, d, cap, _ptr(qb), _ptr(kb), _ptr(vb),
                                    _ptr(idx), _ptr(_i32(count)), max_k, _ptr(out))
    if rc:
        raise ValueError(f"oracle_sparse_attn rc={rc}")
    return out


def evict_step(mode, q, K, V, lens, k, max_k, accum=None, with_attn=True, dtype=None):
    """Whole step.  Returns dict(z, s, accum, idx, count, out, rc)."""
    code = _dtype_code(q, dtype)
    qb, kb, vb = _bits(q), _bits(K), _bits(V)
    B, H, d = qb.shape
    _, Hkv, cap, _ = kb.shape
    z = np.full((B, H, cap), np.nan)
    s = np.full((B, cap), np.nan)
    A = None if accum is None else np.array(accum, dtype=np.float64, copy=True, order="C")
    idx = np.full((B, max_k), -7, dtype=np.int32)
    count = np.zeros(B, dtype=np.int32)
    out = np.zeros((B, H, d)) if with_attn else None
    rc = _load().oracle_evict_step(code, mode, B, H, Hkv, d, cap, _ptr(qb), _ptr(kb), _ptr(vb),
                                   _ptr(_i32(lens)), _ptr(_i32(k)), max_k, _ptr(z), _ptr(s),
                                   _ptr(A), _ptr(idx), _ptr(count), _ptr(out))
    return dict(z=z, s=s, accum=A, idx=idx, count=count, out=out, rc=rc)

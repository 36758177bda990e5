"""The C ABI without a GPU: libhill.so builds, loads and exports every entry
point that include/hill.h declares; host-side validation returns its
documented status before touching the device; the product path never
reaches the oracle and fails loudly without its library."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hill.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2602_18750_gb300 import build, hill
    build.build()
    return hill.load()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hill_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("hill_score", "hill_topk_select", "hill_gather_sparse_attn", "hill_evict_step",
              "hill_topk_select_bkp", "hill_evict_step_bkp", "hill_quantize_k", "hill_score_f8",
              "hill_evict_step_f8", "hill_evict_step_kvh", "hill_selftest_wait",
              "hill_workspace_bytes", "hill_sync_status", "hill_status_string", "hill_abi_version"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2602_18750_gb300 import hill
    out = subprocess.run(["nm", "-D", "--defined-only", hill.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (hill_\w+)", out))
    for n in _declared():
        assert n in exported, f"{n} declared in include/hill.h but not exported"
        assert hasattr(lib, n)


def test_status_strings_and_version(lib):
    from paper_2602_18750_gb300 import hill
    assert lib.hill_abi_version() == 100
    for code, name in [(0, "HILL_OK"), (1, "HILL_ERR_INVALID_ARG"), (2, "HILL_ERR_UNSUPPORTED"),
                       (3, "HILL_ERR_WORKSPACE"), (4, "HILL_ERR_CUDA"), (5, "HILL_ERR_TIMEOUT"),
                       (6, "HILL_ERR_DEVICE")]:
        assert hill.status_string(code) == name


def _desc(**kw):
    from paper_2602_18750_gb300 import hill
    d = dict(batch=2, num_q_heads=8, num_kv_heads=2, head_dim=128, capacity=64, dtype=0,
             q_sb=1024, q_sh=128, k_sb=2 * 64 * 128, k_sh=64 * 128, k_sn=128,
             v_sb=2 * 64 * 128, v_sh=64 * 128, v_sn=128)
    d.update(kw)
    return hill.hill_desc(**d)


FAKE = 1 << 20  # a 16-byte aligned non-null address; validation fails before any access


def _step(lib, desc, **kw):
    a = dict(q=FAKE, k=FAKE, v=FAKE, lens=FAKE, kk=FAKE, max_k=8, mode=0, accum=None, scores=None,
             idx=FAKE, count=FAKE, out=FAKE, ws=FAKE, ws_bytes=1 << 30)
    a.update(kw)
    return lib.hill_evict_step(ctypes.byref(desc) if desc is not None else None, a["q"], a["k"], a["v"],
                               a["lens"], a["kk"], a["max_k"], a["mode"], a["accum"], a["scores"], a["idx"],
                               a["count"], a["out"], a["ws"], a["ws_bytes"], None)


def test_host_validation_without_device(lib):
    from paper_2602_18750_gb300.hill import (HILL_ERR_INVALID_ARG as INV, HILL_ERR_UNSUPPORTED as UNS)
    assert _step(lib, None) == INV
    assert _step(lib, _desc(num_q_heads=6, num_kv_heads=4)) == INV       # H % Hkv
    assert _step(lib, _desc(batch=-1)) == INV
    assert _step(lib, _desc(dtype=7)) == INV
    assert _step(lib, _desc(k_sn=100)) == INV                            # not 16-byte rows
    assert _step(lib, _desc(head_dim=64, q_sh=64)) == UNS
    assert _step(lib, _desc(batch=513)) == UNS                            # above the per-CTA tables
    # any group size and any number of KV heads pass the host checks (the call
    # then fails only for want of a device here)
    from paper_2602_18750_gb300.hill import HILL_ERR_CUDA as CUDA
    for hq, hkv in [(24, 2), (64, 1), (28, 4), (12, 4), (40, 40), (80, 10)]:
        d = _desc(num_q_heads=hq, num_kv_heads=hkv, q_sb=hq * 128,
                  k_sb=hkv * 64 * 128, v_sb=hkv * 64 * 128)
        assert _step(lib, d) == CUDA, (hq, hkv)
    assert _step(lib, _desc(), max_k=-1) == INV
    assert _step(lib, _desc(), q=None) == INV
    assert _step(lib, _desc(), lens=None) == INV
    assert _step(lib, _desc(), idx=None) == INV
    assert _step(lib, _desc(), q=FAKE + 8) == INV                        # misaligned
    assert _step(lib, _desc(), mode=3) == INV
    assert _step(lib, _desc(), v=None) == INV                            # attention needs V
    d = _desc()
    assert lib.hill_score(ctypes.byref(d), FAKE, FAKE, FAKE, 0, None, None, FAKE, 1 << 30, None) == INV
    assert lib.hill_topk_select(ctypes.byref(d), FAKE, FAKE, FAKE, -2, FAKE, FAKE, None, 0, None) == INV
    assert lib.hill_gather_sparse_attn(ctypes.byref(d), FAKE, FAKE, None, FAKE, FAKE, 8, FAKE, None, 0,
                                       None) == INV
    assert lib.hill_workspace_bytes(ctypes.byref(_desc(head_dim=64)), 0, 8) == 0
    # E4M3 shadow: missing or misaligned shadow arrays are rejected before any device work
    assert lib.hill_quantize_k(ctypes.byref(d), FAKE, FAKE, FAKE, 1, None, FAKE, None) == INV
    assert lib.hill_quantize_k(ctypes.byref(d), FAKE, FAKE, FAKE, -1, FAKE, FAKE, None) == INV
    assert lib.hill_score_f8(ctypes.byref(d), FAKE, FAKE + 8, FAKE, FAKE, 0, FAKE, None, FAKE, 1 << 30,
                             None) == INV
    assert lib.hill_evict_step_f8(ctypes.byref(d), FAKE, FAKE, None, None, None, FAKE, FAKE, 8, 0, None, None,
                                  FAKE, FAKE, None, FAKE, 1 << 30, None) == INV
    # per-KV-head step: needs a score or accum buffer; B * Hkv above the attention table is unsupported
    assert lib.hill_evict_step_kvh(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, 8, 0, None, None, FAKE, FAKE,
                                   None, FAKE, 1 << 30, None) == INV
    big = _desc(batch=100, num_q_heads=32, num_kv_heads=8, q_sb=32 * 128)
    assert lib.hill_evict_step_kvh(ctypes.byref(big), FAKE, FAKE, FAKE, FAKE, FAKE, 8, 0, None, FAKE, FAKE, FAKE,
                                   None, FAKE, 1 << 30, None) == UNS
    # BKP: a negative window is rejected before any device work
    assert lib.hill_topk_select_bkp(ctypes.byref(d), FAKE, FAKE, FAKE, -1, 8, FAKE, FAKE, None, None, 0,
                                    None) == INV
    assert lib.hill_evict_step_bkp(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, -1, 8, 0, None, None, FAKE,
                                   FAKE, None, None, FAKE, 1 << 30, None) == INV


def test_binding_fails_loudly_without_library():
    from paper_2602_18750_gb300 import hill
    saved = hill._lib
    hill._lib = None
    try:
        with pytest.raises(OSError):
            hill.load("/nonexistent/libhill.so")
    finally:
        hill._lib = saved


def test_product_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2602_18750_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, flags=re.M), f
                assert "hill_oracle" not in text and "liboracle" not in text, f

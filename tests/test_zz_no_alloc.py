"""hill_score_noalloc: the scoring entry point for callers that cannot
allocate device memory (a plug-in inside a host that owns the device-memory
budget, a latency-critical loop where an allocation could block or fail, a
binding without a CUDA allocator).  Its scratch is a fixed array inside the
library, so it takes no workspace.  Through the C ABI, two calls in a row
must give the same scores as hill_score with a caller-supplied workspace,
within the score tolerance the other parity tests use.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2602_18750_gb300 import inputs

pytestmark = pytest.mark.gpu

RTOL = 1e-3


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2602_18750_gb300 import build, hill
    build.build()
    hill.load()
    return hill


def _close(a, b, lens):
    for i, n in enumerate(lens):
        x, y = a[i, :n].double(), b[i, :n].double()
        floor = y.abs().mean()
        assert torch.all((x - y).abs() <= RTOL * torch.maximum(y.abs(), floor)), f"row {i}"


@pytest.mark.parametrize("heads", [(32, 8), (32, 1)], ids=["gqa", "mqa_dealing"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_noalloc_matches_workspace_call_twice(H, mode, dtype, heads):
    # (32, 1): one KV head with 32 query heads, where the scoring kernel deals
    # the tiles to 8 warps per head, each with its own softmax partial slot
    Hq, Hkv = heads
    lens = [777, 1000, 35]
    q, K, V, lens_t = inputs.random_case(3, Hq, Hkv, 128, 1000, lens, dtype=dtype, seed=17, kind="normal")
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    ws = H.alloc_workspace(desc, mode, 1)
    ref = torch.full((3, 1000), float("nan"), device="cuda")
    H.hill_score(desc, q, K, lens_t, mode, ref, ws=ws)
    lib = H.load()
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        out = torch.full((3, 1000), float("nan"), device="cuda")
        st = lib.hill_score_noalloc(ctypes.byref(desc), q.data_ptr(), K.data_ptr(), lens_t.data_ptr(), mode,
                                    out.data_ptr(), None, stream)
        assert st == H.HILL_OK, H.status_string(st)
        H.hill_sync_status()
        _close(out, ref, lens)


def test_noalloc_accumulates_like_workspace_call(H):
    q, K, V, lens_t = inputs.random_case(2, 8, 8, 128, 300, [300, 211], seed=5, kind="zipf")
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    ws = H.alloc_workspace(desc, 0, 1)
    s_ref, s_new = torch.zeros(2, 300, device="cuda"), torch.zeros(2, 300, device="cuda")
    a_ref, a_new = torch.zeros(2, 300, device="cuda"), torch.zeros(2, 300, device="cuda")
    for _ in range(2):
        H.hill_score(desc, q, K, lens_t, 0, s_ref, a_ref, ws=ws)
        H.hill_score_noalloc(desc, q, K, lens_t, 0, s_new, a_new)
    H.hill_sync_status()
    _close(s_new, s_ref, [300, 211])
    _close(a_new, a_ref, [300, 211])


def test_noalloc_rejects_oversized_call(H):
    # 8 sequences x 32 heads x 32768 tokens of logits (32 MiB) exceed the 16 MiB array
    q = torch.zeros(8, 32, 128, dtype=torch.float16, device="cuda")
    K = torch.zeros(8, 32, 8, 128, dtype=torch.float16, device="cuda")
    desc = H.make_desc(q, K)
    desc.capacity = 32768
    lens = torch.full((8,), 8, dtype=torch.int32, device="cuda")
    out = torch.zeros(8, 8, device="cuda")
    with pytest.raises(H.HillError) as ei:
        H.hill_score_noalloc(desc, q, K, lens, 0, out)
    assert ei.value.status == H.HILL_ERR_WORKSPACE


def _header_limit():
    """HILL_SCORE_NOALLOC_MAX_SCRATCH as include/hill.h defines it."""
    import os
    import re
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    text = open(os.path.join(root, "include", "hill.h")).read()
    m = re.search(r"#define HILL_SCORE_NOALLOC_MAX_SCRATCH \((\d+)u << (\d+)\)", text)
    assert m, "HILL_SCORE_NOALLOC_MAX_SCRATCH not found in include/hill.h"
    return int(m.group(1)) << int(m.group(2))


def _needed_bytes(B, Hq, Hkv, cap, sms):
    """Scratch of an ATTN call as include/hill.h states it: logits, softmax
    partials and statistics, each rounded up to 256 bytes."""
    W = 8 // Hkv if (Hkv <= 4 and Hq // Hkv >= 5) else 1
    P = min(sms, B * ((cap + 31) // 32)) * W
    r = lambda x: (x + 255) // 256 * 256
    return r(4 * B * Hq * cap) + r(8 * B * Hq * P) + r(8 * B * Hq)


@pytest.mark.parametrize("heads", [(32, 8), (32, 1)], ids=["gqa", "mqa_dealing"])
def test_noalloc_size_limit_is_the_stated_formula(H, heads):
    """The largest capacity whose stated scratch fits the array is accepted
    (and scores like hill_score); 32 tokens more is rejected."""
    Hq, Hkv = heads
    limit = _header_limit()
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    cap = 32
    while _needed_bytes(1, Hq, Hkv, cap + 32, sms) <= limit:
        cap += 32
    assert _needed_bytes(1, Hq, Hkv, cap + 32, sms) > limit
    lens = [300]
    q, K, V, lens_t = inputs.random_case(1, Hq, Hkv, 128, 300, lens, seed=23, kind="zipf")
    Kbig = torch.zeros(1, Hkv, cap + 32, 128, dtype=K.dtype, device="cuda")
    Kbig[:, :, :300] = K.cuda()
    q, lens_t = q.cuda(), lens_t.cuda()
    for c, ok in ((cap, True), (cap + 32, False)):
        Kc = Kbig[:, :, :c]
        desc = H.make_desc(q, Kc)
        out = torch.full((1, c), float("nan"), device="cuda")
        if not ok:
            with pytest.raises(H.HillError) as ei:
                H.hill_score_noalloc(desc, q, Kc, lens_t, 0, out)
            assert ei.value.status == H.HILL_ERR_WORKSPACE
            continue
        H.hill_score_noalloc(desc, q, Kc, lens_t, 0, out)
        ref = torch.full((1, c), float("nan"), device="cuda")
        H.hill_score(desc, q, Kc, lens_t, 0, ref, ws=H.alloc_workspace(desc, 0, 1))
        H.hill_sync_status()
        _close(out, ref, lens)

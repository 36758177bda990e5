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


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("dtype", [torch.float16, torch.bfloat16])
def test_noalloc_matches_workspace_call_twice(H, mode, dtype):
    lens = [777, 1000, 35]
    q, K, V, lens_t = inputs.random_case(3, 32, 8, 128, 1000, lens, dtype=dtype, seed=17, kind="normal")
    q, K, lens_t = q.cuda(), K.cuda(), lens_t.cuda()
    desc = H.make_desc(q, K)
    ws = H.alloc_workspace(desc, mode, 1)
    ref = torch.zeros(3, 1000, device="cuda")
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

"""cast_route_topk_noalloc: routing for callers that cannot allocate device memory.

Some callers (plugins inside a framework that owns every device allocation, real-time loops
that must not enter an allocator, fixed-budget runtimes) cannot hand the library a workspace.
The allocation-free entry point uses the library's own fixed 16 MiB device array instead.
These tests call it through the C ABI twice in a row and compare each result with the
allocating entry point's on the same inputs; they also check that a problem needing more
scratch than the fixed array is refused with a clear message.  The file name makes pytest
collect it last, and it passes both alone in a fresh process and after the other tests.
"""
import ctypes as C

import numpy as np
import pytest
import torch

from synthetic import generators as G
from tests.gpu_util import to_dev, to_host

pytestmark = pytest.mark.gpu


def _inputs(seed, N=3, S=300, H=4, d=128, M=12, Bv=200):
    ss = np.random.SeedSequence(seed)
    a, b, c = ss.spawn(3)
    q = G.round_bf16(G.tokens_with_offsets(a, N, S, H, d, 1.0))
    k = G.round_bf16(G.tokens_with_offsets(b, M, Bv, H, d, 1.0))
    v = G.round_bf16(G.tokens_with_offsets(c, M, Bv, H, d, 1.0))
    return to_dev(q, "bf16"), to_dev(k, "bf16"), to_dev(v, "bf16")


def _call_noalloc(lib, q, anchors, k, v, K, refine=None):
    """Direct C-ABI call of cast_route_topk_noalloc (no workspace argument)."""
    a = lib._route_args(q, anchors, k, v, K, refine=refine)
    Kf, H, M = len(anchors), q.shape[2], k.shape[0]
    idx = torch.full((Kf, H, min(K, M)), -1, dtype=torch.int32, device="cuda")
    u = torch.full((Kf, H, M), float("nan"), dtype=torch.float32, device="cuda")
    a.idx, a.u = C.c_void_p(idx.data_ptr()), C.c_void_p(u.data_ptr())
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    status = lib.library().cast_route_topk_noalloc(C.byref(a), stream)
    assert status == lib.OK, lib.library().cast_last_error_detail()
    return idx, u


def test_noalloc_matches_workspace_entry_point_twice(lib):
    anchors, K = [0, 2], 3
    for call, seed in enumerate((31, 32)):
        q, k, v = _inputs(seed)
        ref_idx, ref_u = lib.cast_route_topk(q, anchors, k, v, K, want_u=True)
        idx, u = _call_noalloc(lib, q, anchors, k, v, K)
        torch.cuda.synchronize()
        np.testing.assert_allclose(to_host(u), to_host(ref_u), rtol=2e-4, atol=1e-7)
        assert np.array_equal(idx.cpu().numpy(), ref_idx.cpu().numpy()), f"call {call}"


def test_noalloc_wide_path_with_refinement(lib):
    """Many history blocks (the per-head statistics spread over a cluster of CTAs, radix-select
    TopK) with the paper's two refinement passes: the shared scratch is left holding another
    problem's means by the call before, and each result must still equal the workspace entry
    point's."""
    anchors, K, M = [0, 2, 4, 6], 90, 448
    for call, seed in enumerate((41, 42)):
        q, k, v = _inputs(seed, N=8, S=40, H=2, d=128, M=M, Bv=16)
        # a different problem through the fixed scratch first
        q0, k0, v0 = _inputs(seed + 100)
        _call_noalloc(lib, q0, [0, 1], k0, v0, 5, refine=lib.REFINE_PAPER)
        ref_idx, ref_u = lib.cast_route_topk(q, anchors, k, v, K, want_u=True, refine=lib.REFINE_PAPER)
        idx, u = _call_noalloc(lib, q, anchors, k, v, K, refine=lib.REFINE_PAPER)
        torch.cuda.synchronize()
        lib.cast_check_device()
        np.testing.assert_allclose(to_host(u), to_host(ref_u), rtol=2e-4, atol=1e-7)
        assert np.array_equal(idx.cpu().numpy(), ref_idx.cpu().numpy()), f"call {call}"


def test_noalloc_rejects_problems_above_its_fixed_scratch(lib):
    # the f32 means of 2 anchor frames and 600 key and value blocks of 32 heads x 128 channels
    # (19.7 MB) exceed 16 MiB
    q = torch.zeros((2, 64, 32, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((600, 64, 32, 128), dtype=torch.bfloat16, device="cuda")
    a = lib._route_args(q, [0, 1], k, k, 4)
    assert lib.library().cast_route_workspace_size(C.byref(a)) > (16 << 20)
    idx = torch.empty((2, 32, 4), dtype=torch.int32, device="cuda")
    a.idx = C.c_void_p(idx.data_ptr())
    status = lib.library().cast_route_topk_noalloc(C.byref(a), None)
    assert status == lib.ERR_UNSUPPORTED
    assert b"16 MiB" in lib.library().cast_last_error_detail()

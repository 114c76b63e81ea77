"""Paper-granularity history blocks (App. C Tab. config: (t, h, w) = (1, 8, 8) in token
coordinates, partial blocks masked; Tab. config_cast: K = ceil(0.2 M)): routing, routed
attention and the block step over history frames [F_h, Hg, Wg, H, d], against the oracle fed
the same frames cut by its own `spatial_blocks`."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import ATTN_REL_MAX, to_dev, to_host
from tests.test_gpu_block_step import _check, _run_block
from tests.test_gpu_refine import check_refined
from tests.test_gpu_route import check_idx

pytestmark = pytest.mark.gpu


def _frames(seed, F, Hg, Wg, H, d, dtype="bf16", off=1.0):
    a, b = np.random.SeedSequence(seed).spawn(2)
    k = G.frames_with_region_offsets(a, F, Hg, Wg, H, d, off)
    v = G.frames_with_region_offsets(b, F, Hg, Wg, H, d, off)
    if dtype == "bf16":
        k, v = G.round_bf16(k), G.round_bf16(v)
    return k, v


def _blocks(x):
    """[F, Hg, Wg, H, d] -> the oracle's list of (1, 8, 8) blocks [n_m, H, d]."""
    F, Hg, Wg, H, d = x.shape
    return O.gather_blocks(x.reshape(F, Hg * Wg, H, d), O.spatial_blocks(F, Hg, Wg))


def _cur(seed, N, S, H, d, dtype="bf16"):
    parts = np.random.SeedSequence(seed).spawn(3)
    out = [G.tokens_with_offsets(p, N, S, H, d, 0.5) for p in parts]
    return [G.round_bf16(x) for x in out] if dtype == "bf16" else out


ROUTE_CASES = [
    # F_h, Hg, Wg, H, d, dtype
    (3, 11, 13, 2, 64, "bf16"),      # 2 x 2 blocks per frame, three of them truncated
    (2, 16, 24, 3, 128, "f32"),      # only full blocks
    (4, 30, 52, 2, 128, "bf16"),     # the Matrix-Game grid: 4 x 7 blocks, 10 truncated
    (1, 5, 3, 1, 64, "bf16"),        # one block of 15 tokens
]


@pytest.mark.parametrize("case", ROUTE_CASES, ids=lambda c: f"F{c[0]}_{c[1]}x{c[2]}_H{c[3]}d{c[4]}_{c[5]}")
def test_route_spatial_blocks(lib, case):
    F, Hg, Wg, H, d, dtype = case
    N, anchors = 3, [0, 2]
    q = _cur(40 + Hg, N, Hg * Wg, H, d, dtype)[0]
    kf, vf = _frames(41 + Wg, F, Hg, Wg, H, d, dtype)
    kl, vl = _blocks(kf), _blocks(vf)
    M = len(kl)
    K = O.paper_budget(M)
    idx, u, (qb, kb, vb) = lib.cast_route_topk(to_dev(q, dtype), anchors, to_dev(kf, dtype),
                                                to_dev(vf, dtype), K, want_u=True, want_pooled=True)
    torch.cuda.synchronize()
    assert idx.shape == (len(anchors), H, min(K, M))
    rt = O.pooled_routing(q, anchors, kl, vl)
    np.testing.assert_allclose(to_host(qb), rt.qbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(kb), rt.kbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(vb), rt.vbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(u), rt.u, rtol=2e-4, atol=1e-7 * rt.u.max())
    check_idx(idx.cpu().numpy(), rt.u, min(K, M))


def test_route_spatial_refined(lib):
    """Coupled refinement (Alg. routing, the paper's 2 passes) over (1, 8, 8) blocks."""
    F, Hg, Wg, H, d = 3, 30, 52, 2, 128
    N, anchors = 8, [0, 2, 4, 6]
    q = _cur(50, N, Hg * Wg, H, d)[0]
    kf, vf = _frames(51, F, Hg, Wg, H, d)
    kl, vl = _blocks(kf), _blocks(vf)
    K = O.paper_budget(len(kl))
    idx, u = lib.cast_route_topk(to_dev(q, "bf16"), anchors, to_dev(kf, "bf16"), to_dev(vf, "bf16"),
                                 K, want_u=True, refine=lib.REFINE_PAPER)
    torch.cuda.synchronize()
    rt = O.pooled_routing(q, anchors, kl, vl)
    ug = to_host(u)
    np.testing.assert_allclose(ug, rt.u, rtol=2e-4, atol=1e-7 * rt.u.max())
    # the oracle's refinement on the GPU's own omission scores (exact outside ambiguous heads)
    check_refined(idx.cpu().numpy(), ug, anchors, N, K, lib.REFINE_PAPER)


ATTN_CASES = [
    # N, Hg, Wg, H, d, F_h, K, anchors, out dtype
    (3, 11, 13, 2, 64, 3, 5, (0, 2), torch.float32),       # odd K: last tile half empty
    (2, 16, 24, 2, 128, 2, 4, (1,), torch.bfloat16),       # full blocks only
    (2, 30, 52, 2, 128, 4, 23, (0, 1), torch.float32),     # K = ceil(0.2 * 112)
    (2, 9, 9, 1, 128, 2, 1, (0,), torch.float32),          # one routed block
]


@pytest.mark.parametrize("case", ATTN_CASES, ids=lambda c: f"N{c[0]}_{c[1]}x{c[2]}_H{c[3]}d{c[4]}_F{c[5]}K{c[6]}")
def test_attention_spatial_blocks(lib, case):
    N, Hg, Wg, H, d, F, K, anchors, odt = case
    S = Hg * Wg
    q, kc, vc = _cur(60 + d + Hg, N, S, H, d)
    kf, vf = _frames(61 + Wg, F, Hg, Wg, H, d)
    kl, vl = _blocks(kf), _blocks(vf)
    M = len(kl)
    rng = np.random.default_rng(S + K)
    # every (anchor, head) routes the last (bottom-right, truncated in both directions) block
    # plus random others, in an arbitrary order
    idx = np.stack([[np.concatenate([[M - 1], rng.permutation(M - 1)[:K - 1]])[rng.permutation(K)]
                     for _ in range(H)] for _ in anchors]).astype(np.int32)
    dk = (lambda x: to_dev(x, "bf16"))
    o, lse = lib.cast_anchor_attention(dk(q), dk(kc), dk(vc), list(anchors), dk(kf), dk(vf),
                                       torch.from_numpy(idx).cuda(), out_dtype=odt, want_lse=True)
    torch.cuda.synchronize()
    lib.cast_check_device()
    ref, lse_ref = O.routed_attention(q, kc, vc, kl, vl, list(anchors), idx, with_lse=True)
    ref = ref.reshape(len(anchors), S, H * d)
    err = float(np.max(np.abs(to_host(o) - ref)) / np.max(np.abs(ref)))
    assert err <= ATTN_REL_MAX, err
    np.testing.assert_allclose(to_host(lse), lse_ref, atol=2e-2)


def test_attention_spatial_all_blocks_is_dense(lib):
    """Routing every (1, 8, 8) block equals dense attention over the chunk and every history
    token: masking drops exactly the positions outside the grid."""
    N, Hg, Wg, H, d, F = 2, 13, 11, 2, 128, 2
    S = Hg * Wg
    q, kc, vc = _cur(70, N, S, H, d)
    kf, vf = _frames(71, F, Hg, Wg, H, d)
    M = len(O.spatial_blocks(F, Hg, Wg))
    idx = np.tile(np.arange(M, dtype=np.int32), (1, H, 1))
    dk = (lambda x: to_dev(x, "bf16"))
    o = lib.cast_anchor_attention(dk(q), dk(kc), dk(vc), [1], dk(kf), dk(vf),
                                  torch.from_numpy(np.ascontiguousarray(idx)).cuda(),
                                  out_dtype=torch.float32)
    torch.cuda.synchronize()
    # dense reference: the history frames as one block holding all F * S tokens
    dense = [kf.reshape(F * S, H, d)], [vf.reshape(F * S, H, d)]
    ref = O.routed_attention(q, kc, vc, dense[0], dense[1], [1], np.zeros((1, H, 1), np.int64))
    err = float(np.max(np.abs(to_host(o) - ref.reshape(1, S, H * d))) / np.max(np.abs(ref)))
    assert err <= ATTN_REL_MAX, err


TINY64 = W.BlockStepWorkload("tiny64_f32_4f_12x10_h2d64_hist2f_m8_k2", 8, 4, (12, 10), 2, 64, 8, 64,
                             2, (0, 3), "f32", band_radius=2.0, hist_frames=2)


def _oracle_inputs(inp):
    return dict(inp, k_hist=_blocks(inp["k_hist"]), v_hist=_blocks(inp["v_hist"]))


def test_block_step_spatial_tiny(lib):
    wl = TINY64
    inp = W.block_step_inputs(wl)
    assert inp["k_hist"].shape == (2, 12, 10, 2, 64)
    out = _run_block(lib, wl, inp, with_x=True)
    _check(wl, _oracle_inputs(inp), out)
    np.testing.assert_allclose(out["x"], out["x0"] + out["r"], rtol=1e-6, atol=1e-6)


def test_block_step_spatial_full_size(lib):
    """The Matrix-Game shape at the paper's granularity: 16 history frames = 448 blocks,
    K = 90; routed blocks, a sample of attention rows and PAR tiles against the oracle."""
    wl = W.MG64
    inp = W.block_step_inputs(wl)
    out = _run_block(lib, wl, inp)
    rng = np.random.default_rng(wl.seed)
    rows = np.unique(np.concatenate([[0, wl.S - 1], rng.integers(0, wl.S, 6)]))
    ntile = len(O.tiles_of(wl.grid[0], wl.grid[1], 8, 8))
    tiles = sorted({0, ntile - 1, int(rng.integers(0, ntile))})
    _check(wl, _oracle_inputs(inp), out, rows=rows, tiles=tiles)

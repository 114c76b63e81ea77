"""cast_block_step (route -> attention -> PAR) against the oracle, stage by stage: each stage
is compared with the oracle fed the GPU's own upstream result, so errors do not compound."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import workloads as W
from tests.gpu_util import ATTN_REL_MAX, par_check, to_dev, to_host
from tests.test_gpu_route import check_idx

pytestmark = pytest.mark.gpu


def _run_block(lib, wl, inp, with_x=False, refine=None):
    dk = (lambda x: to_dev(x, "bf16"))
    N, S, H, d = inp["q"].shape
    rdt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    r_out = torch.zeros((N, S, H * d), dtype=rdt, device="cuda")
    keff = min(wl.K, wl.M)
    idx = torch.empty((len(wl.anchors), H, keff), dtype=torch.int32, device="cuda")
    x = None
    if with_x:
        x = torch.randn((N, S, H * d), generator=torch.Generator().manual_seed(0)).to(rdt).cuda()
        x0 = x.clone()
    params = lib.par_params(band_radius=wl.band_radius)
    lib.cast_block_step(dk(inp["q"]), dk(inp["k_cur"]), dk(inp["v_cur"]), list(wl.anchors),
                        dk(inp["k_hist"]), dk(inp["v_hist"]), wl.K, wl.grid, r_out, x=x,
                        idx_out=idx, params=params, refine=refine)
    torch.cuda.synchronize()
    lib.cast_check_device()
    out = {"r": to_host(r_out), "idx": idx.cpu().numpy()}
    if with_x:
        out["x"], out["x0"] = to_host(x), to_host(x0)
    return out


def _check(wl, inp, out, rows=None, tiles=None, routing=True):
    anchors = list(wl.anchors)
    Kf = len(anchors)
    N, S, H, d = inp["q"].shape
    # routing
    if routing:
        rt = O.pooled_routing(inp["q"], anchors, inp["k_hist"], inp["v_hist"])
        check_idx(out["idx"], rt.u, min(wl.K, wl.M))
    # attention, fed the GPU's routed blocks
    ref = O.routed_attention(inp["q"], inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                             anchors, out["idx"], rows=rows)
    sel = slice(None) if rows is None else rows
    g = out["r"][anchors].reshape(Kf, S, H, d)[:, sel]
    r = ref[:, sel]
    assert np.max(np.abs(g - r)) / np.max(np.abs(r)) <= ATTN_REL_MAX
    # PAR, fed the GPU's anchor rows
    mask = W.anchor_mask(N, anchors)
    R = np.zeros((N, wl.grid[0], wl.grid[1], H * d))
    R[anchors] = out["r"][anchors].reshape(Kf, wl.grid[0], wl.grid[1], H * d)
    p = O.ParParams(band_radius=wl.band_radius)
    pref, info = O.par_reconstruct(R, mask, None, p, tiles=tiles, with_info=True)
    tiles_all = O.tiles_of(wl.grid[0], wl.grid[1], 8, 8)
    amb = [(tiles_all[ti][0], tiles_all[ti][2]) for (ti, a, b), tt in info.items()
           if tt.branch_ambiguous or tt.threshold_ambiguous]
    gp = out["r"].reshape(N, wl.grid[0], wl.grid[1], H * d)
    targets = [t for t in range(N) if not mask[t]]
    if tiles is None:
        par_check(gp, pref, targets, wl.dtype, excluded_tiles=amb)
    else:
        for ti in tiles:
            y0, h, x0, w = tiles_all[ti]
            if (y0, x0) in amb:
                continue
            par_check(gp[:, y0:y0 + h, x0:x0 + w], pref[:, y0:y0 + h, x0:x0 + w], targets, wl.dtype)


def test_block_step_tiny(lib):
    wl = W.TINY
    inp = W.block_step_inputs(wl)
    out = _run_block(lib, wl, inp, with_x=True)
    _check(wl, inp, out)
    np.testing.assert_allclose(out["x"], out["x0"] + out["r"], rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("wl", [W.MG, W.HY], ids=lambda w: w.name)
def test_block_step_full_size(lib, wl):
    inp = W.block_step_inputs(wl)
    out = _run_block(lib, wl, inp)
    rng = np.random.default_rng(wl.seed)
    rows = np.unique(np.concatenate([[0, wl.S - 1], rng.integers(0, wl.S, 6)]))
    ntile = len(O.tiles_of(wl.grid[0], wl.grid[1], 8, 8))
    tiles = sorted({0, ntile - 1, int(rng.integers(0, ntile)), int(rng.integers(0, ntile))})
    _check(wl, inp, out, rows=rows, tiles=tiles)


DEGENERATE = [
    # every frame an anchor: PAR has nothing to reconstruct, every row is attention output
    W.BlockStepWorkload("all_anchors_f32_3f_12x10_h2d64_m3_k2", 11, 3, (12, 10), 2, 64, 3, 40, 2,
                        (0, 1, 2), "f32"),
    # budget above the history: every block routed (TopK bypassed), bf16 residual
    W.BlockStepWorkload("bypass_bf16_5f_9x13_h2d128_m3_k7", 12, 5, (9, 13), 2, 128, 3, 70, 7,
                        (0, 4), "bf16"),
    # one anchor pair in the middle: frames on both sides extrapolated (alpha < 0 and > 1),
    # tiles of sides 8, 3 and 1
    W.BlockStepWorkload("extrap_f32_6f_11x9_h1d64_m5_k2", 13, 6, (11, 9), 1, 64, 5, 33, 2,
                        (2, 3), "f32"),
]


@pytest.mark.parametrize("wl", DEGENERATE, ids=lambda w: w.name)
def test_block_step_degenerate(lib, wl):
    inp = W.block_step_inputs(wl)
    out = _run_block(lib, wl, inp)
    if wl.K >= wl.M:
        assert np.array_equal(out["idx"], np.tile(np.arange(wl.M, dtype=np.int32),
                                                  (len(wl.anchors), wl.H, 1)))
    _check(wl, inp, out)


@pytest.mark.parametrize("wl", [W.MG, W.HY], ids=lambda w: w.name)
def test_block_step_refined_full_size(lib, wl):
    """The bench configurations: the Matrix-Game- and HY-World-shaped block steps with the
    paper's two refinement passes (Alg. routing).  The omission scores are compared with the
    oracle's, the refined block sets with Alg. routing run by the oracle on those scores, and
    the attention rows and PAR outputs with the oracle fed the GPU's routed blocks / anchor
    rows (sampled rows on both sides of query-tile boundaries, the first and last tile pair
    included; every tile shape of the grid)."""
    from tests.test_gpu_par_configs import edge_kind_sample
    from tests.test_gpu_refine import PAPER, check_refined
    inp = W.block_step_inputs(wl)
    out = _run_block(lib, wl, inp, refine=PAPER)
    anchors = list(wl.anchors)
    dk = (lambda x: to_dev(x, "bf16"))
    _, u = lib.cast_route_topk(dk(inp["q"]), anchors, dk(inp["k_hist"]), dk(inp["v_hist"]), wl.K,
                               want_u=True, refine=PAPER)
    torch.cuda.synchronize()
    ug = to_host(u)
    rt = O.pooled_routing(inp["q"], anchors, inp["k_hist"], inp["v_hist"])
    np.testing.assert_allclose(ug, rt.u, rtol=1e-3, atol=1e-6 * rt.u.max())
    changed, amb = check_refined(out["idx"], ug, anchors, wl.n_cur, wl.K, PAPER)
    assert amb < wl.H
    rng = np.random.default_rng(wl.seed + 1)
    last = wl.S - wl.S % 256 if wl.S % 256 else wl.S - 256   # first row of the last tile pair
    bounds = [0, 127, 128, 255, 256, last - 1, last, last + 127, last + 128, wl.S - 1]
    rows = np.unique(np.concatenate([[b for b in bounds if 0 <= b < wl.S], rng.integers(0, wl.S, 4)]))
    ntile = len(O.tiles_of(wl.grid[0], wl.grid[1], 8, 8))
    tiles = edge_kind_sample(wl.grid[0], wl.grid[1], extra=(int(rng.integers(0, ntile)),))
    _check(wl, inp, out, rows=rows, tiles=tiles, routing=False)

"""The residual sites beyond the attention output: the block step with the output projection
W_O (PAR on the post-projection residual), and the anchor FFN site (cast_ffn_step), against
the oracle stage by stage (each stage fed the GPU's own upstream result)."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import ATTN_REL_MAX, par_check, to_dev, to_host

pytestmark = pytest.mark.gpu


def _rel_err(gpu, ref):
    return float(np.max(np.abs(gpu - ref)) / np.max(np.abs(ref)))


def _par_stage(r_gpu, anchors, N, grid, C, dtype, band=-1.0, wch=None):
    """PAR of the oracle fed the GPU's anchor rows, checked on every skipped frame."""
    mask = W.anchor_mask(N, anchors)
    R = np.zeros((N, grid[0], grid[1], C))
    R[anchors] = r_gpu.reshape(N, grid[0], grid[1], C)[anchors]
    p = O.ParParams(band_radius=band)
    ref, info = O.par_reconstruct(R, mask, wch, p, with_info=True)
    tiles_all = O.tiles_of(grid[0], grid[1], 8, 8)
    amb = [(tiles_all[ti][0], tiles_all[ti][2]) for (ti, a, b), tt in info.items()
           if tt.branch_ambiguous or tt.threshold_ambiguous]
    targets = [t for t in range(N) if not mask[t]]
    par_check(r_gpu.reshape(N, grid[0], grid[1], C), ref, targets, dtype, excluded_tiles=amb)


def _weights(seed, D_out, D_in, bias_dtype):
    ss = np.random.SeedSequence(seed)
    a, b = ss.spawn(2)
    w = G.round_bf16(G.normal(a, (D_out, D_in), 1.0 / np.sqrt(D_in)))
    bias = G.normal(b, (D_out,), 0.1)
    if bias_dtype == "bf16":
        bias = G.round_bf16(bias)
    return w, bias


@pytest.mark.parametrize("wl,with_bias", [(W.TINY, True), (W.TINY, False), (W.MG, True)],
                         ids=["tiny_bias", "tiny_nobias", "mg_bias"])
def test_block_step_output_projection(lib, wl, with_bias):
    inp = W.block_step_inputs(wl)
    N, S, H, d = inp["q"].shape
    D = H * d
    anchors = list(wl.anchors)
    w_o, b_o = _weights(40 + N, D, D, wl.dtype)
    dk = (lambda x: to_dev(x, "bf16"))
    rdt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    r_out = torch.zeros((N, S, D), dtype=rdt, device="cuda")
    idx = torch.empty((len(anchors), H, min(wl.K, wl.M)), dtype=torch.int32, device="cuda")
    lib.cast_block_step(dk(inp["q"]), dk(inp["k_cur"]), dk(inp["v_cur"]), anchors,
                        dk(inp["k_hist"]), dk(inp["v_hist"]), wl.K, wl.grid, r_out, idx_out=idx,
                        params=lib.par_params(band_radius=wl.band_radius),
                        w_o=dk(w_o), b_o=to_dev(b_o, wl.dtype) if with_bias else None)
    torch.cuda.synchronize()
    lib.cast_check_device()
    r = to_host(r_out)
    idx_h = idx.cpu().numpy()
    # attention fed the GPU's routing, then the projection of the oracle's attention output
    rows = None if wl is W.TINY else np.unique(np.r_[0, S - 1, np.random.default_rng(3).integers(0, S, 6)])
    Oref = O.routed_attention(inp["q"], inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                              anchors, idx_h, rows=rows)
    for i, a in enumerate(anchors):
        o_rows = Oref[i] if rows is None else Oref[i][rows]
        ref = O.linear(o_rows.reshape(-1, D), w_o, b_o if with_bias else None)
        got = r[a] if rows is None else r[a][rows]
        assert _rel_err(got, ref) <= ATTN_REL_MAX
    if wl is W.TINY:
        _par_stage(r, anchors, N, wl.grid, D, wl.dtype, wl.band_radius)


FFN_CASES = [
    # F, grid, D, D_ff, anchors, r dtype
    (6, (11, 13), 64, 256, (1, 3), "f32"),
    (7, (9, 16), 128, 512, (0, 2, 5), "bf16"),
    # K not a multiple of the 64-wide k-slice, N not a multiple of the 32-column epilogue chunk
    # nor of the 256-column tile, 17 x 9 = 153 rows (a ragged second row tile), three anchors
    (5, (17, 9), 72, 200, (0, 2, 4), "f32"),
]


@pytest.mark.parametrize("case", FFN_CASES, ids=lambda c: f"F{c[0]}_{c[1][0]}x{c[1][1]}_D{c[2]}_{c[5]}")
def test_ffn_step_small(lib, case):
    F, grid, D, Dff, anchors, rdt = case
    S = grid[0] * grid[1]
    ss = np.random.SeedSequence(F * 7 + D)
    x = G.round_bf16(G.normal(ss, (F, S, D)))
    w1, b1 = _weights(1 + D, Dff, D, "bf16")
    w2, b2 = _weights(2 + D, D, Dff, rdt)
    tdt = torch.float32 if rdt == "f32" else torch.bfloat16
    r_out = torch.zeros((F, S, D), dtype=tdt, device="cuda")
    lib.cast_ffn_step(to_dev(x, "bf16"), list(anchors), to_dev(w1, "bf16"), to_dev(b1, "bf16"),
                      to_dev(w2, "bf16"), to_dev(b2, rdt), grid, r_out)
    torch.cuda.synchronize()
    lib.cast_check_device()
    r = to_host(r_out)
    ref = O.anchor_ffn(x, list(anchors), w1, b1, w2, b2)
    for i, a in enumerate(anchors):
        assert _rel_err(r[a], ref[i]) <= ATTN_REL_MAX
    _par_stage(r, list(anchors), F, grid, D, rdt)


def test_ffn_step_matrix_game_size(lib):
    """The Matrix-Game-shaped site: 8 frames of 30x52, D = 1536, D_ff = 6144, anchors every
    second frame, bf16 residual; anchor rows sampled, PAR on sampled tiles."""
    wl = W.MG
    N, S, D, Dff = wl.n_cur, wl.S, wl.H * wl.d, 4 * wl.H * wl.d
    anchors = list(wl.anchors)
    x = G.round_bf16(G.normal(np.random.SeedSequence(91), (N, S, D)))
    w1, b1 = _weights(92, Dff, D, "bf16")
    w2, b2 = _weights(93, D, Dff, "bf16")
    r_out = torch.zeros((N, S, D), dtype=torch.bfloat16, device="cuda")
    lib.cast_ffn_step(to_dev(x, "bf16"), anchors, to_dev(w1, "bf16"), to_dev(b1, "bf16"),
                      to_dev(w2, "bf16"), to_dev(b2, "bf16"), wl.grid, r_out)
    torch.cuda.synchronize()
    lib.cast_check_device()
    r = to_host(r_out)
    rows = np.unique(np.r_[0, S - 1, np.random.default_rng(5).integers(0, S, 6)])
    for a in anchors:
        hid = O.gelu_tanh(O.linear(x[a][rows], w1, b1))
        ref = O.linear(hid, w2, b2)
        assert _rel_err(r[a][rows], ref) <= ATTN_REL_MAX
    # PAR fed the GPU's anchor rows, on a few tiles
    mask = W.anchor_mask(N, anchors)
    R = np.zeros((N, wl.grid[0], wl.grid[1], D))
    R[anchors] = r.reshape(N, wl.grid[0], wl.grid[1], D)[anchors]
    tiles_all = O.tiles_of(wl.grid[0], wl.grid[1], 8, 8)
    tiles = [0, len(tiles_all) - 1, 9]
    pref, info = O.par_reconstruct(R, mask, None, O.ParParams(), tiles=tiles, with_info=True)
    amb = {ti for (ti, _, _), tt in info.items() if tt.branch_ambiguous or tt.threshold_ambiguous}
    gp = r.reshape(N, wl.grid[0], wl.grid[1], D)
    targets = [t for t in range(N) if not mask[t]]
    for ti in tiles:
        if ti in amb:
            continue
        y0, h, x0, w = tiles_all[ti]
        par_check(gp[:, y0:y0 + h, x0:x0 + w], pref[:, y0:y0 + h, x0:x0 + w], targets, "bf16")

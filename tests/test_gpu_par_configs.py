"""PAR on the block-step configurations' own residual inputs, against the oracle.

The residuals are the ones the configurations define (Section 4.3, App. A.2 Eq.
exacttranslation is the regime they exercise): the tiny case's N(0,1) frame rolled by t
tokens plus 0.05 noise, and Gaussian random fields (correlation length 4 tokens) under
per-frame 0-3 token camera shifts for the Matrix-Game- and HY-World-shaped chunks (the
latter with 1 % amplitude drift per frame).  Coherent translations give reliable bins,
confidence near one and a gate near one at low frequencies, so the phase transport does real
work here.  Every tile is compared for the tiny and Matrix-Game shapes, a sample holding the
first, last and every kind of edge tile for the HY-World shape; f32 within 1e-4 of the frame
RMS, bf16 within that plus the output rounding.  Tiles the oracle flags as branch- or
threshold-ambiguous are excluded and counted (at most 1 %).
"""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import par_check, to_dev, to_host

pytestmark = pytest.mark.gpu


def edge_kind_sample(Hg, Wg, extra=()):
    """Tile indices: first, last, one of every (h, w) tile shape of the grid, plus extra."""
    tiles = O.tiles_of(Hg, Wg, 8, 8)
    pick = {0, len(tiles) - 1, *extra}
    seen = set()
    for ti, (y0, h, x0, w) in enumerate(tiles):
        if (h, w) not in seen:
            seen.add((h, w))
            pick.add(ti)
    return sorted(pick)


def _run_and_check(lib, wl, R, dtype, tiles):
    N = wl.n_cur
    mask = W.anchor_mask(N, wl.anchors)
    r = to_dev(R, dtype)
    params = lib.par_params(band_radius=wl.band_radius)
    lib.cast_par_reconstruct(r, mask, None, params)
    torch.cuda.synchronize()
    lib.cast_check_device()
    gpu = to_host(r)
    Rin = G.round_bf16(R) if dtype == "bf16" else R
    p = O.ParParams(band_radius=wl.band_radius)
    ref, info = O.par_reconstruct(Rin, mask, None, p, tiles=tiles, with_info=True)
    tiles_all = O.tiles_of(wl.grid[0], wl.grid[1], 8, 8)
    n_checked = len(tiles_all) if tiles is None else len(tiles)
    amb = sorted({(tiles_all[ti][0], tiles_all[ti][2]) for (ti, a, b), tt in info.items()
                  if tt.branch_ambiguous or tt.threshold_ambiguous})
    print(f"{wl.name} {dtype}: {len(amb)} ambiguous of {n_checked} tiles")
    assert len(amb) <= max(1, n_checked // 100)
    targets = [t for t in range(N) if not mask[t]]
    sel = range(len(tiles_all)) if tiles is None else tiles
    for ti in sel:
        y0, h, x0, w = tiles_all[ti]
        if (y0, x0) in amb:
            continue
        par_check(gpu[:, y0:y0 + h, x0:x0 + w], ref[:, y0:y0 + h, x0:x0 + w], targets, dtype)
    for a in wl.anchors:   # anchors untouched
        src = G.round_bf16(R[a]) if dtype == "bf16" else R[a]
        assert np.array_equal(gpu[a], src.astype(np.float64))
    return info


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("wl", [W.TINY, W.MG], ids=lambda w: w.name)
def test_par_config_residuals_every_tile(lib, wl, dtype):
    R = W.par_residuals(wl)
    info = _run_and_check(lib, wl, R, dtype, None)
    # translating content: the pooled confidence of most (tile, pair) transports is high
    conf = [tt.c for tt in info.values()]
    assert np.median(conf) > 0.5, np.median(conf)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_par_config_residuals_hy_sampled(lib, dtype):
    wl = W.HY
    R = W.par_residuals(wl)
    tiles = edge_kind_sample(wl.grid[0], wl.grid[1], extra=(9, 23, 37))
    _run_and_check(lib, wl, R, dtype, tiles)

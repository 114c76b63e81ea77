"""PAR kernel (cast_par_reconstruct) against the CPU oracle, element by element."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import par_check, to_dev, to_host

pytestmark = pytest.mark.gpu


def _ambiguous_tiles(info, tiles_all):
    out = []
    for (ti, a, b), tt in info.items():
        if tt.branch_ambiguous or tt.threshold_ambiguous:
            y0, h, x0, w = tiles_all[ti]
            out.append((y0, x0))
    return out


def _run(lib, R, mask, dtype, wch=None, **pp):
    r = to_dev(R, dtype)
    wt = None if wch is None else torch.from_numpy(wch.astype(np.float32)).cuda()
    params = lib.par_params(**{k: v for k, v in pp.items() if k != "gate"},
                            gate_mode={"paper": lib.GATE_PAPER, "zero": lib.GATE_ZERO,
                                       "one": lib.GATE_ONE}[pp.get("gate", "paper")])
    lib.cast_par_reconstruct(r, mask, wt, params)
    torch.cuda.synchronize()
    return to_host(r)


def _oracle(R, mask, dtype, wch=None, tiles=None, **pp):
    Rin = G.round_bf16(R) if dtype == "bf16" else R
    p = O.ParParams(tile_h=pp.get("tile", (8, 8))[0], tile_w=pp.get("tile", (8, 8))[1],
                    band_radius=pp.get("band_radius", -1.0), gate_mode=pp.get("gate", "paper"))
    ref, info = O.par_reconstruct(Rin, mask, wch, p, tiles=tiles, with_info=True)
    return ref, info, p


CASES = [
    # F, Hg, Wg, C, anchors, dtype, extra
    (6, 11, 13, 40, (1, 3), "f32", {}),
    (6, 11, 13, 40, (1, 3), "bf16", {}),
    (7, 17, 20, 264, (0, 2, 5), "f32", {}),
    (7, 17, 20, 264, (0, 2, 5), "f32", {"gate": "zero"}),
    (7, 17, 20, 264, (0, 2, 5), "f32", {"gate": "one"}),
    (7, 17, 20, 264, (0, 2, 5), "f32", {"band_radius": 2.0}),
    (5, 9, 9, 128, (2, 4), "f32", {"tile": (4, 6)}),
    (9, 8, 8, 136, (0, 8), "f32", {}),
    (9, 8, 8, 136, (0, 8), "bf16", {"band_radius": 4.0}),
    # one tile and three anchor pairs (one time segment per pair); 1096 channels: 9 channel
    # chunks of 128, the last one partly empty
    (8, 8, 8, 1096, (0, 2, 5, 7), "f32", {}),
    # 4096 channels: 32 chunks
    (5, 16, 24, 4096, (0, 4), "bf16", {}),
    # edge tiles of sides 7 and 2 (15 = 8 + 7 rows, 10 = 8 + 2 columns)
    (5, 15, 10, 72, (0, 3), "f32", {}),
    # edge tiles of sides 6 and 4 (the Matrix-Game remainders), frame 0 extrapolated
    (5, 14, 12, 48, (1, 4), "bf16", {}),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"F{c[0]}_{c[1]}x{c[2]}_C{c[3]}_{c[5]}_{c[6]}")
def test_par_small(lib, case):
    F, Hg, Wg, Cc, anchors, dtype, extra = case
    R, _ = G.grf_sequence(np.random.SeedSequence([F, Hg, Wg, Cc]), F, Hg, Wg, Cc, ell=3.0)
    R += 0.1 * np.random.default_rng(1).standard_normal(R.shape).astype(np.float32)
    mask = W.anchor_mask(F, anchors)
    wch = np.random.default_rng(2).uniform(0, 1, Cc).astype(np.float32) if Cc == 264 else None
    gpu = _run(lib, R, mask, dtype, wch, **extra)
    ref, info, p = _oracle(R, mask, dtype, wch, **extra)
    tiles_all = O.tiles_of(Hg, Wg, p.tile_h, p.tile_w)
    amb = _ambiguous_tiles(info, tiles_all)
    assert len(amb) <= max(1, len(tiles_all) // 100)
    targets = [t for t in range(F) if not mask[t]]
    par_check(gpu, ref, targets, dtype, excluded_tiles=amb, th=p.tile_h, tw=p.tile_w)
    # anchor frames untouched
    for a in anchors:
        src = G.round_bf16(R[a]) if dtype == "bf16" else R[a]
        assert np.array_equal(gpu[a], src.astype(np.float64))


def test_par_all_anchors_is_noop(lib):
    R = np.random.default_rng(3).standard_normal((3, 8, 8, 16)).astype(np.float32)
    gpu = _run(lib, R, [1, 1, 1], "f32")
    assert np.array_equal(gpu, R.astype(np.float64))


def test_par_rejects_single_anchor(lib):
    r = torch.zeros((3, 8, 8, 16), device="cuda")
    with pytest.raises(lib.CastError) as e:
        lib.cast_par_reconstruct(r, [0, 1, 0])
    assert e.value.status == lib.ERR_INVALID_ARG


def test_par_translation_identity(lib):
    """g = 1 on a band-limited circular shift reconstructs the phase-interpolated shift."""
    rng = np.random.default_rng(4)
    Fx = np.fft.rfft2(rng.standard_normal((16, 8, 8)), norm="ortho")
    Fx[:, :, 2:] = 0
    base = np.fft.irfft2(Fx, s=(8, 8), norm="ortho").transpose(1, 2, 0)
    R = np.zeros((3, 8, 8, 16), dtype=np.float32)
    R[0] = base
    R[2] = np.roll(base, 2, axis=1)
    gpu = _run(lib, R, [1, 0, 1], "f32", gate="one")
    np.testing.assert_allclose(gpu[1], np.roll(base, 1, axis=1), atol=2e-5)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("spacing", [2, 3, 4])
def test_par_sweep_full_size_sampled(lib, dtype, spacing):
    """The PAR sweep workload [16, 44, 80, 3072] at full size, weights U[0,1], band 4:
    every output of a sample of tiles (interior and ragged edge) against the oracle."""
    w = W.PAR_SWEEP
    R, wch = W.par_sweep_inputs(w)
    anchors = w.anchors(spacing)
    mask = W.anchor_mask(w.F, anchors)
    gpu = _run(lib, R, mask, dtype, wch, band_radius=w.band_radius)
    tiles_all = O.tiles_of(w.grid[0], w.grid[1], 8, 8)
    sample = [0, 7, 23, 49, 50, 55, 59]   # last row (50..59) has 4-token-high edge tiles
    ref, info, _ = _oracle(R, mask, dtype, wch, tiles=sample, band_radius=w.band_radius)
    amb = _ambiguous_tiles(info, tiles_all)
    assert len(amb) <= 1
    targets = [t for t in range(w.F) if not mask[t]]
    for ti in sample:
        y0, h, x0, ww = tiles_all[ti]
        if (y0, x0) in amb:
            continue
        sl = (slice(y0, y0 + h), slice(x0, x0 + ww))
        par_check(gpu[:, sl[0], sl[1]], ref[:, sl[0], sl[1]], targets, dtype)


def test_par_tensor_core_blend_edge_shapes(lib):
    """bf16 with enough (tile, 128-channel chunk) items per tile kind that both the full 8x8
    tiles and the truncated edge tiles (8x4 right column, 6x8 bottom row, 6x4 corner of a 30x52
    grid) take the tensor-core blend; one pair carries five targets (two stacked groups and a
    single), frames 5 and 6 extrapolated.  Every output of the edge tiles and of two full tiles
    against the oracle."""
    F, Hg, Wg, Cc, anchors = 7, 30, 52, 4096, (0, 4)
    R, _ = G.grf_sequence(np.random.SeedSequence([F, Hg, Wg, Cc, 7]), F, Hg, Wg, Cc, ell=3.0)
    mask = W.anchor_mask(F, anchors)
    gpu = _run(lib, R, mask, "bf16")
    tiles_all = O.tiles_of(Hg, Wg, 8, 8)
    sample = [i for i, (y0, h, x0, w) in enumerate(tiles_all) if h < 8 or w < 8] + [0, 8]
    ref, info, _ = _oracle(R, mask, "bf16", tiles=sample)
    amb = _ambiguous_tiles(info, tiles_all)
    assert len(amb) <= 1
    targets = [t for t in range(F) if not mask[t]]
    for ti in sample:
        y0, h, x0, w = tiles_all[ti]
        if (y0, x0) in amb:
            continue
        sl = (slice(y0, y0 + h), slice(x0, x0 + w))
        par_check(gpu[:, sl[0], sl[1]], ref[:, sl[0], sl[1]], targets, "bf16")

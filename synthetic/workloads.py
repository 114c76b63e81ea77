"""The five synthetic workloads (shapes, anchors, budgets, seeds) and their input builders.

Shapes follow the paper's two backbones (Section 5.1, Tab. config,
Tab. config_cast): chunk-autoregressive latent video with token grids per frame,
frame-sized historical KV blocks, a per-anchor historical budget K and 8x8 PAR
tiles.  Inputs are seeded draws from `synthetic.generators`; bf16 workloads are
rounded to bf16 here so that every consumer sees identical bits.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from . import generators as G


@dataclass(frozen=True)
class BlockStepWorkload:
    name: str
    seed: int
    n_cur: int            # current latent frames N_cur
    grid: tuple           # (Hg, Wg); S = Hg * Wg tokens per frame
    H: int                # heads
    d: int                # head dim
    M: int                # history blocks
    B_v: int              # tokens per history block
    K: int                # routing budget K_KV
    anchors: tuple        # ascending anchor frame indices
    dtype: str            # "bf16" or "f32" (residual/output dtype)
    band_radius: float = -1.0   # < 0: no band cut (the paper's gate on every bin)
    offset_scale: float = 1.0   # per-(frame|block, head) offsets of the tokens
    amp_drift: float = 0.0      # per-frame amplitude drift of the PAR residual fields
    hist_frames: int = 0        # > 0: the history is this many frames of the chunk's grid,
                                # cut into (1, 8, 8) blocks (M of them, B_v = 64 nominal)

    @property
    def S(self):
        return self.grid[0] * self.grid[1]

    @property
    def D(self):
        return self.H * self.d


TINY = BlockStepWorkload("tiny_f32_4f_8x8_h2d64_m4_k2", 0, 4, (8, 8), 2, 64, 4, 64, 2,
                         (0, 3), "f32", band_radius=2.0, offset_scale=0.0)
MG = BlockStepWorkload("mg_bf16_8f_30x52_h12d128_m16_k4", 1, 8, (30, 52), 12, 128, 16, 1560,
                       4, (0, 2, 4, 6), "bf16")
HY = BlockStepWorkload("hy_bf16_16f_44x80_h24d128_m32_k8", 2, 16, (44, 80), 24, 128, 32, 3520,
                       8, (0, 3, 7, 12, 15), "bf16", amp_drift=0.01)


# The paper's KV granularity (App. C Tab. config: (1, 8, 8) blocks, partial blocks masked;
# Tab. config_cast: K = ceil(0.2 M)) on the two backbone shapes with 16 / 32 history frames:
# 30x52 tokens = 4 x 7 blocks per frame, 44x80 = 6 x 10.
MG64 = BlockStepWorkload("mg64_bf16_8f_30x52_h12d128_hist16f_m448_k90", 6, 8, (30, 52), 12, 128,
                         448, 64, 90, (0, 2, 4, 6), "bf16", hist_frames=16)
HY64 = BlockStepWorkload("hy64_bf16_16f_44x80_h24d128_hist32f_m1920_k384", 7, 16, (44, 80), 24, 128,
                         1920, 64, 384, (0, 3, 7, 12, 15), "bf16", amp_drift=0.01, hist_frames=32)


@dataclass(frozen=True)
class StressWorkload:
    name: str = "stress_bf16_4f_44x80_h24d128_m128"
    seed: int = 4
    n_cur: int = 4
    grid: tuple = (44, 80)
    H: int = 24
    d: int = 128
    M: int = 128
    B_v: int = 3520
    Ks: tuple = (4, 8, 16, 32)
    n_planted: int = 8

    @property
    def S(self):
        return self.grid[0] * self.grid[1]


STRESS = StressWorkload()


@dataclass(frozen=True)
class ParSweepWorkload:
    name: str = "par_sweep_16f_44x80_c3072"
    seed: int = 3
    F: int = 16
    grid: tuple = (44, 80)
    C: int = 3072
    spacings: tuple = (2, 3, 4)
    band_radius: float = 4.0
    dtypes: tuple = ("f32", "bf16")

    def anchors(self, spacing):
        return tuple(range(0, self.F, spacing))


PAR_SWEEP = ParSweepWorkload()


def anchor_mask(n_frames, anchors):
    m = np.zeros(n_frames, dtype=np.uint8)
    m[list(anchors)] = 1
    return m


# --------------------------------------------------------------------------
# builders
# --------------------------------------------------------------------------


def _maybe_bf16(x, dtype):
    return G.round_bf16(x) if dtype == "bf16" else x


def block_step_inputs(w: BlockStepWorkload, scale_rows: int | None = None):
    """Inputs of one block step: q, k_cur, v_cur [N_cur, S, H, d], k_hist, v_hist
    [M, B_v, H, d] (or history frames [F_h, Hg, Wg, H, d] when w.hist_frames) (float32 holding
    bf16 values: the attention runs in bf16),
    plus anchors and the mask.  All current frames carry Q (only anchor rows
    are read)."""
    ss = np.random.SeedSequence(w.seed)
    sq, skc, svc, skh, svh = ss.spawn(5)
    S = w.S
    q = G.tokens_with_offsets(sq, w.n_cur, S, w.H, w.d, w.offset_scale)
    kc = G.tokens_with_offsets(skc, w.n_cur, S, w.H, w.d, w.offset_scale)
    vc = G.tokens_with_offsets(svc, w.n_cur, S, w.H, w.d, w.offset_scale)
    if w.hist_frames:
        # history frames [F_h, Hg, Wg, H, d]; (1, 8, 8) blocks carry their own offsets
        Hg, Wg = w.grid
        kh = G.frames_with_region_offsets(skh, w.hist_frames, Hg, Wg, w.H, w.d, w.offset_scale)
        vh = G.frames_with_region_offsets(svh, w.hist_frames, Hg, Wg, w.H, w.d, w.offset_scale)
    else:
        kh = G.tokens_with_offsets(skh, w.M, w.B_v, w.H, w.d, w.offset_scale)
        vh = G.tokens_with_offsets(svh, w.M, w.B_v, w.H, w.d, w.offset_scale)
    out = dict(q=q, k_cur=kc, v_cur=vc, k_hist=kh, v_hist=vh)
    for k in out:
        out[k] = G.round_bf16(out[k])
    out["anchors"] = np.asarray(w.anchors, dtype=np.int32)
    out["anchor_mask"] = anchor_mask(w.n_cur, w.anchors)
    return out


def par_residuals(w: BlockStepWorkload):
    """Standalone PAR residuals of a block-step workload, [N_cur, Hg, Wg, D].

    TINY: an N(0,1) frame rolled by t tokens along W plus 0.05 N(0,1) noise.
    MG/HY: Gaussian random fields (correlation length 4 tokens) under a
    per-frame 0-3 token camera shift (HY adds 1 % amplitude drift per frame)."""
    ss = np.random.SeedSequence([w.seed, 7])
    Hg, Wg = w.grid
    if w is TINY or w.name.startswith("tiny"):
        r = G.shifted_noise_sequence(ss, w.n_cur, Hg, Wg, w.D, noise=0.05)
    else:
        r, _ = G.grf_sequence(ss, w.n_cur, Hg, Wg, w.D, ell=4.0, max_shift=3,
                              amp_drift=w.amp_drift)
    return _maybe_bf16(r, w.dtype)


def par_sweep_inputs(w: ParSweepWorkload = PAR_SWEEP):
    """GRF residuals [F, Hg, Wg, C] (float32) and per-channel weights U[0,1)."""
    ss = np.random.SeedSequence(w.seed)
    s_r, s_w = ss.spawn(2)
    r, _ = G.grf_sequence(s_r, w.F, w.grid[0], w.grid[1], w.C, ell=4.0, max_shift=3)
    wc = G.uniform_weights(s_w, w.C)
    return r, wc


def stress_inputs(w: StressWorkload = STRESS):
    """Long-history stress: every current frame is an anchor; anchor queries carry
    the per-head direction g_h that 8 planted history blocks share."""
    ss = np.random.SeedSequence(w.seed)
    sq, skc, svc, shist = ss.spawn(4)
    S = w.S
    g, planted, kh, vh = G.planted_history(shist, w.M, w.B_v, w.H, w.d, w.n_planted)
    q = G.normal(sq, (w.n_cur, S, w.H, w.d))
    q += g[None, None, :, :]
    kc = G.normal(skc, (w.n_cur, S, w.H, w.d))
    vc = G.normal(svc, (w.n_cur, S, w.H, w.d))
    out = dict(q=q, k_cur=kc, v_cur=vc, k_hist=kh, v_hist=vh)
    for k in out:
        out[k] = G.round_bf16(out[k])
    out["anchors"] = np.arange(w.n_cur, dtype=np.int32)
    out["anchor_mask"] = np.ones(w.n_cur, dtype=np.uint8)
    out["planted"] = planted
    return out


@dataclass(frozen=True)
class SelectWorkload:
    """Control-aware frame selection at a block of the Matrix-Game-shaped chunk: two control
    branches (camera, action) of [N_cur, S, D] bf16 updates, K_f of N_cur frames."""
    name: str = "select_mg_bf16_8f_30x52_c1536_k4"
    seed: int = 5
    n_cur: int = 8
    grid: tuple = (30, 52)
    D: int = 1536
    n_branch: int = 2
    K_f: int = 4


SELECT_MG = SelectWorkload()


def select_inputs(w: SelectWorkload = SELECT_MG):
    """bf16-rounded control updates, refresh ages and the previous block's anchor mask."""
    ss = np.random.SeedSequence(w.seed)
    sd, sa = ss.spawn(2)
    S = w.grid[0] * w.grid[1]
    deltas = [G.round_bf16(x) for x in G.control_updates(sd, w.n_branch, w.n_cur, S, w.D)]
    rng = G._gen(sa)
    ages = rng.integers(0, 4, w.n_cur).astype(np.int32)
    mask = np.zeros(w.n_cur, dtype=np.uint8)
    mask[rng.choice(w.n_cur, w.K_f, replace=False)] = 1
    return deltas, ages, mask

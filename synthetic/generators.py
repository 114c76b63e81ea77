"""Seeded synthetic inputs shared by the CPU oracle checks and the CUDA path.

This module holds no arithmetic of the method itself: it draws random numbers
(numpy PCG64, fixed draw order), rounds them to the exact bf16 bits the GPU
receives, and shapes them like the paper's workloads (Section 5.1,
Tab. config: latent token grids, 8x8 spectral tiles, frame-sized history
blocks).  Both the oracle and the GPU path consume the arrays produced here.
"""
from __future__ import annotations

import concurrent.futures as _cf
import os

import numpy as np
import scipy.ndimage as _nd

# --------------------------------------------------------------------------
# bf16 helpers (round-to-nearest-even, the rounding of a cvt.rn.bf16.f32)
# --------------------------------------------------------------------------


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 array -> uint16 bf16 bit patterns, round-to-nearest-even."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """uint16 bf16 bit patterns -> float32 values (exact)."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """float32 values rounded to the nearest bf16 value, returned as float32."""
    return bf16_to_f32(bf16_bits(x))


# --------------------------------------------------------------------------
# parallel seeded normal draws
# --------------------------------------------------------------------------

_CHUNK = 1 << 22


def normal(seed_seq: np.random.SeedSequence, shape, scale: float = 1.0) -> np.ndarray:
    """N(0, scale^2) float32 array of `shape`.

    The flat array is cut into fixed 4 Mi-element chunks, chunk k drawn from
    the k-th child of `seed_seq`; the result depends only on the seed and the
    shape, not on the thread count."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.float32)
    nchunks = (n + _CHUNK - 1) // _CHUNK
    children = seed_seq.spawn(nchunks)

    def fill(k):
        lo, hi = k * _CHUNK, min(n, (k + 1) * _CHUNK)
        np.random.Generator(np.random.PCG64(children[k])).standard_normal(
            out=out[lo:hi], dtype=np.float32)

    if nchunks == 1:
        fill(0)
    else:
        workers = min(nchunks, max(1, (os.cpu_count() or 1)))
        with _cf.ThreadPoolExecutor(workers) as ex:
            list(ex.map(fill, range(nchunks)))
    if scale != 1.0:
        out *= np.float32(scale)
    return out.reshape(shape)


def _gen(seed_seq: np.random.SeedSequence) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed_seq))


# --------------------------------------------------------------------------
# token tensors for routing / attention
# --------------------------------------------------------------------------


def tokens_with_offsets(seed_seq, n_groups: int, rows: int, H: int, d: int,
                        offset_scale: float) -> np.ndarray:
    """[n_groups, rows, H, d] float32: N(0,1) tokens plus one N(0, offset_scale^2)
    d-vector per (group, head) added to every token of the group.

    Groups are frames (queries / current K,V) or history blocks; the offsets
    make pooled means spread O(1) so that routing scores are not all ties."""
    s_tok, s_off = seed_seq.spawn(2)
    x = normal(s_tok, (n_groups, rows, H, d))
    if offset_scale:
        off = _gen(s_off).standard_normal((n_groups, 1, H, d), dtype=np.float32)
        x += np.float32(offset_scale) * off
    return x


def frames_with_region_offsets(seed_seq, n_frames: int, Hg: int, Wg: int, H: int, d: int,
                               offset_scale: float, region: int = 8) -> np.ndarray:
    """[n_frames, Hg, Wg, H, d] float32 history frames: N(0,1) tokens plus one
    N(0, offset_scale^2) d-vector per (frame, region x region patch of the token grid, head),
    so that the means of neighbouring patches differ by O(1).  Patches at the right and
    bottom edges are cut by the grid."""
    s_tok, s_off = seed_seq.spawn(2)
    x = normal(s_tok, (n_frames, Hg, Wg, H, d))
    if offset_scale:
        ny, nx = -(-Hg // region), -(-Wg // region)
        off = _gen(s_off).standard_normal((n_frames, ny, nx, H, d), dtype=np.float32)
        off = np.repeat(np.repeat(off, region, axis=1), region, axis=2)[:, :Hg, :Wg]
        x += np.float32(offset_scale) * off
    return x


# --------------------------------------------------------------------------
# residual fields for PAR
# --------------------------------------------------------------------------


def grf_sequence(seed_seq, F: int, Hg: int, Wg: int, C: int, ell: float = 4.0,
                 max_shift: int = 3, amp_drift: float = 0.0):
    """Gaussian-random-field residuals [F, Hg, Wg, C] float32 seen by a panning camera.

    Per channel, white N(0,1) noise on a canvas of (Hg + s*F) x (Wg + s*F)
    (s = max_shift) is smoothed with a Gaussian of std ell/sqrt(2) (field
    covariance ~ exp(-r^2 / 2 ell^2), correlation length ell tokens) and
    renormalised to unit variance.  Frame t is the crop at the cumulative
    offset sum_{tau<=t} delta_tau with delta_tau uniform in {0..s}^2
    (delta_0 = 0), scaled by (1 + amp_drift)^t.  Returns (frames, offsets)."""
    s_noise, s_shift = seed_seq.spawn(2)
    pad = max_shift * F
    canvas = normal(s_noise, (Hg + pad, Wg + pad, C))
    sig = ell / np.sqrt(2.0)
    canvas = _nd.gaussian_filter(canvas, sigma=(sig, sig, 0), mode="wrap")
    canvas /= np.float32(canvas.std())
    steps = _gen(s_shift).integers(0, max_shift + 1, size=(F, 2))
    steps[0] = 0
    offs = np.cumsum(steps, axis=0)
    out = np.empty((F, Hg, Wg, C), dtype=np.float32)
    for t in range(F):
        oy, ox = offs[t]
        out[t] = canvas[oy:oy + Hg, ox:ox + Wg, :]
        if amp_drift:
            out[t] *= np.float32((1.0 + amp_drift) ** t)
    return out, offs


def shifted_noise_sequence(seed_seq, F: int, Hg: int, Wg: int, C: int,
                           noise: float = 0.05) -> np.ndarray:
    """R_0 ~ N(0,1) [Hg, Wg, C]; R_t = roll(R_0, t tokens along W) + noise*N(0,1)."""
    s0, s1 = seed_seq.spawn(2)
    r0 = normal(s0, (Hg, Wg, C))
    eps = normal(s1, (F, Hg, Wg, C), scale=noise)
    out = np.empty((F, Hg, Wg, C), dtype=np.float32)
    for t in range(F):
        out[t] = np.roll(r0, t, axis=1) + (eps[t] if t else 0.0)
    return out


def uniform_weights(seed_seq, C: int) -> np.ndarray:
    """Per-channel confidence weights uniform in [0, 1)."""
    return _gen(seed_seq).random(C, dtype=np.float32)


def planted_history(seed_seq, M: int, B_v: int, H: int, d: int, n_planted: int = 8):
    """Long-history keys/values with planted high-similarity blocks.

    Returns (g, planted, k_hist, v_hist): g [H, d] ~ N(0, I) per head; for each
    head, `n_planted` distinct blocks (planted[h, j]) get K += beta_j g_h with
    beta_j = 0.25 (1 + j/7); every other block gets K += N(0, 0.25^2) d-vector;
    every block gets V += an N(0,1) d-vector."""
    s_g, s_pick, s_k, s_v, s_koff, s_voff = seed_seq.spawn(6)
    g = _gen(s_g).standard_normal((H, d), dtype=np.float32)
    pick = _gen(s_pick)
    planted = np.stack([pick.permutation(M)[:n_planted] for _ in range(H)])
    k = normal(s_k, (M, B_v, H, d))
    v = normal(s_v, (M, B_v, H, d))
    koff = _gen(s_koff).standard_normal((M, H, d), dtype=np.float32) * np.float32(0.25)
    for h in range(H):
        for j, m in enumerate(planted[h]):
            koff[m, h] = np.float32(0.25 * (1.0 + j / 7.0)) * g[h]
    k += koff[:, None, :, :]
    v += _gen(s_voff).standard_normal((M, 1, H, d), dtype=np.float32)
    return g, planted, k, v


def control_updates(seed_seq, n_branch: int, N: int, S: int, D: int, lo: float = 0.2,
                    hi: float = 2.0):
    """Control-branch feature updates: n_branch arrays [N, S, D] float32, frame i of branch k
    drawn N(0, a_{k,i}^2) with amplitudes a_{k,i} ~ U[lo, hi) so the frames' response
    magnitudes differ (the conditioning-path updates of camera / action branches)."""
    out = []
    for child in seed_seq.spawn(n_branch):
        ca, cn = child.spawn(2)
        amp = _gen(ca).uniform(lo, hi, N).astype(np.float32)
        x = normal(cn, (N, S, D))
        x *= amp[:, None, None]
        out.append(x)
    return out

"""CPU oracle of CAST's per-block anchor/skip step: routing, routed anchor attention, PAR.

TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and the cpu_baseline /
reference leg of bench.py may import this module.  The library's product path
never calls it, and it shares no code with the CUDA path.

Everything is float64 numpy written as the paper states it: the DFT is its
defining double sum (as products with the DFT matrices), the softmax is
explicit, TopK is a full sort.  Inputs are the exact values the GPU receives
(bf16-rounded where the GPU reads bf16).

Readings of points where the paper is silent, ambiguous or garbled:
  * pooled statistics are arithmetic means over tokens (Eq. pooled);
  * eps in Eq. (omission) is 1e-8 (the paper's stated epsilon of App. A.2);
  * TopK ties go to the lower block index; the selected set is returned ascending;
  * a tile's conjugate pairs in the kx = 0 and kx = w/2 columns take the phase
    and the reliability decided at their representative (0 < ky < h/2), the
    mirror gets the negated phase; self-conjugate bins get U = 1 (App. A.2);
  * theta = Arg Z in (-pi, pi]  (a computed -pi is mapped to +pi);
  * nu = r / r_max with r = sqrt((ky_signed/h)^2 + (kx/w)^2), r_max over the
    tile's stored bins (App. A.2, "largest represented radius");
  * optional band cut: bins with rho = sqrt((ky_s*8/h)^2 + (kx*8/w)^2) > band
    radius get g = 0 (plain interpolation); band < 0 is the paper's gate;
  * optional per-channel weights w_c >= 0 multiply both pooled sums of Eq. (cross).

Parity unpinned: the full paper gate of PAR on data that is not a translation.  The
paper prints no worked example for it; the pins fix its pieces (the transform, the
confidence bounds and closed forms, the gate's limits g = 0 / g = 1, exact translations
and Prop. 1) and one property of the whole (time reversal: swapping a pair's anchors with
alpha -> 1 - alpha reconstructs the same frames), and beyond them the oracle is the
definition itself.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

# ===========================================================================
# Section 4.3 / App. A.2: orthonormal 2-D real DFT of a tile, per channel
# ===========================================================================


def dft_matrix(n: int, sign: int) -> np.ndarray:
    """E[k, j] = exp(sign * 2 pi i k j / n)."""
    k = np.arange(n)
    return np.exp(sign * 2j * np.pi * np.outer(k, k) / n)


def rfft2_ortho(x: np.ndarray) -> np.ndarray:
    """x [..., h, w] real -> F [..., h, w//2 + 1],
    F[ky, kx] = (h w)^(-1/2) sum_y sum_x x[y, x] exp(-2 pi i (ky y / h + kx x / w))."""
    h, w = x.shape[-2:]
    ey = dft_matrix(h, -1)                      # [ky, y]
    ex = dft_matrix(w, -1)[:, : w // 2 + 1]     # [x, kx]
    return (ey @ x @ ex) / np.sqrt(h * w)


def hermitian_full(F: np.ndarray, w: int) -> np.ndarray:
    """Half spectrum [..., h, w//2+1] -> full [..., h, w] using F(ky, kx) = conj F(-ky, -kx)."""
    h = F.shape[-2]
    wr = w // 2 + 1
    full = np.zeros(F.shape[:-2] + (h, w), dtype=complex)
    full[..., :, :wr] = F
    neg_ky = (-np.arange(h)) % h
    for kx in range(wr, w):
        full[..., :, kx] = np.conj(F[..., neg_ky, w - kx])
    return full


def irfft2_ortho(F: np.ndarray, w: int, check: bool = True) -> np.ndarray:
    """Inverse of rfft2_ortho: full Hermitian spectrum, full complex inverse DFT, real part.
    With check=True the imaginary part must vanish (real-valuedness, App. A.2)."""
    h = F.shape[-2]
    full = hermitian_full(F, w)
    x = (dft_matrix(h, +1) @ full @ dft_matrix(w, +1)) / np.sqrt(h * w)
    if check:
        scale = max(float(np.sqrt(np.mean(x.real ** 2))), 1e-300)
        assert float(np.max(np.abs(x.imag))) <= 1e-9 * scale + 1e-300, "non-Hermitian spectrum"
    return x.real


# ===========================================================================
# Bin bookkeeping of an (h, w) tile's stored half spectrum (App. A.2)
# ===========================================================================


@dataclass
class TileBins:
    h: int
    w: int
    kappa: np.ndarray        # [h, wr] multiplicity of the real FFT (1 or 2)
    selfconj: np.ndarray     # [h, wr] bool: self-conjugate bins (U = 1)
    rep: np.ndarray          # [h, wr, 2] (ky, kx) of the representative of each bin
    mirror: np.ndarray       # [h, wr] bool: bin whose phase is minus its representative's
    dc: np.ndarray           # [h, wr] bool
    nu: np.ndarray           # [h, wr] normalized radial frequency in [0, 1]
    rho: np.ndarray          # [h, wr] radius in 8x8-tile bin units (band cut)


def tile_bins(h: int, w: int) -> TileBins:
    wr = w // 2 + 1
    ky, kx = np.meshgrid(np.arange(h), np.arange(wr), indexing="ij")
    edge_col = (kx == 0) | ((w % 2 == 0) & (kx == w // 2))
    kappa = np.where(edge_col, 1, 2)
    half_row = (ky == 0) | ((h % 2 == 0) & (ky == h // 2))
    selfconj = edge_col & half_row
    mirror = edge_col & ~selfconj & (ky > h / 2)
    rep = np.stack([np.where(mirror, (h - ky) % h, ky), kx], axis=-1)
    dc = (ky == 0) & (kx == 0)
    ky_s = np.where(ky <= (h - 1) // 2, ky, ky - h)           # numpy fftfreq convention
    r = np.sqrt((ky_s / h) ** 2 + (kx / w) ** 2)
    rmax = r.max()
    nu = r / rmax if rmax > 0 else np.zeros_like(r)
    rho = np.sqrt((ky_s * 8.0 / h) ** 2 + (kx * 8.0 / w) ** 2)
    return TileBins(h, w, kappa, selfconj, rep, mirror, dc, nu, rho)


# ===========================================================================
# Phase-Aware Reconstruction (Section 4.3; App. A.2)
# ===========================================================================


@dataclass
class ParParams:
    """Defaults from Tab. config_cast and App. A.2."""
    tile_h: int = 8
    tile_w: int = 8
    tau_low: float = 0.25
    tau_high: float = 0.75
    q: float = 2.0
    T: float = 0.10
    eps: float = 1e-8
    eta_rel: float = 1e-6
    eta_abs: float = 1e-8
    band_radius: float = -1.0
    gate_mode: str = "paper"     # "paper" | "zero" (g = 0) | "one" (g = 1)


@dataclass
class TileTransport:
    Z: np.ndarray
    W: np.ndarray
    eta: float
    reliable: np.ndarray   # [h, wr] after propagation to mirrors
    theta: np.ndarray      # [h, wr] phase of U (0 where U = 1)
    c: float
    g: np.ndarray          # [h, wr]
    branch_ambiguous: bool
    threshold_ambiguous: bool


def tile_transport(Fa: np.ndarray, Fb: np.ndarray, wch, p: ParParams, bins: TileBins,
                   amb_tol: float = 1e-5) -> TileTransport:
    """Pooled cross-spectrum, reliability, principal phase, tile confidence and gate.

    Fa, Fb: [C, h, wr] spectra of the two anchors.  Eqs. (cross), (confidence),
    (gate) and the numerical conventions of App. A.2."""
    wc = np.ones(Fa.shape[0]) if wch is None else np.asarray(wch, dtype=np.float64)
    Z = np.einsum("c,cij->ij", wc, Fb * np.conj(Fa))              # Eq. (cross)
    W = np.einsum("c,cij->ij", wc, np.abs(Fb) * np.abs(Fa))
    eta = p.eta_rel * W.max() + p.eta_abs                          # App. A.2 threshold
    Zabs = np.abs(Z)
    rel_bin = (W > eta) & (Zabs > eta)
    ry, rx = bins.rep[..., 0], bins.rep[..., 1]
    reliable = rel_bin[ry, rx]                                     # decided at the representative
    theta_rep = np.angle(Z[ry, rx])                                # principal branch
    theta_rep = np.where(theta_rep <= -np.pi, np.pi, theta_rep)    # (-pi, pi]
    theta = np.where(bins.mirror, -theta_rep, theta_rep)
    theta = np.where(reliable & ~bins.selfconj, theta, 0.0)        # U = 1 elsewhere
    omega_plus = reliable & ~bins.dc                               # reliable non-DC bins
    if omega_plus.any():
        c = float(np.sum(bins.kappa * Zabs * omega_plus) /
                  (np.sum(bins.kappa * W * omega_plus) + p.eps))   # Eq. (confidence)
    else:
        c = 0.0
        theta = np.zeros_like(theta)
    tau = p.tau_low + (p.tau_high - p.tau_low) * bins.nu ** p.q     # Eq. (gate)
    g = 1.0 / (1.0 + np.exp(-(c - tau) / p.T))
    if p.gate_mode == "zero":
        g = np.zeros_like(g)
    elif p.gate_mode == "one":
        g = np.ones_like(g)
    if p.band_radius >= 0:
        g = np.where(bins.rho > p.band_radius, 0.0, g)
    # ambiguity flags: results jump when theta crosses +-pi or a bin crosses eta
    rep_bins = reliable & ~bins.selfconj & ~bins.mirror
    branch_amb = bool(np.any(rep_bins & (np.pi - np.abs(theta_rep) < amb_tol)))
    thr_amb = bool(np.any(np.abs(W - eta) <= amb_tol * eta) or
                   np.any(np.abs(Zabs - eta) <= amb_tol * eta))
    return TileTransport(Z, W, eta, reliable, theta, c, g, branch_amb, thr_amb)


def blend(Fa, Fb, theta, g, alpha):
    """Eq. (fcpasm): F_t = (1-a) F_a U^{g a} + a F_b U^{-g (1-a)}, U^b = exp(i b theta)."""
    return ((1.0 - alpha) * Fa * np.exp(1j * g * alpha * theta) +
            alpha * Fb * np.exp(-1j * g * (1.0 - alpha) * theta))


def skipped_assignment(anchor_mask):
    """Eq. (block): every skipped frame t -> (a, b, alpha).  Interior frames use their
    bracketing anchors, frames before a_0 use (a_0, a_1), frames after a_J use
    (a_{J-1}, a_J); alpha = (t - a) / (b - a) (negative / above 1 at the boundary)."""
    mask = np.asarray(anchor_mask).astype(bool)
    anchors = np.flatnonzero(mask)
    F = mask.size
    if anchors.size == F:
        return []
    if anchors.size < 2:
        raise ValueError("PAR needs at least two anchors when a frame is skipped")
    out = []
    for t in range(F):
        if mask[t]:
            continue
        if t < anchors[0]:
            a, b = anchors[0], anchors[1]
        elif t > anchors[-1]:
            a, b = anchors[-2], anchors[-1]
        else:
            a = anchors[anchors < t].max()
            b = anchors[anchors > t].min()
        out.append((t, int(a), int(b), (t - a) / (b - a)))
    return out


def tiles_of(Hg, Wg, th, tw):
    """Disjoint tiles anchored at (0, 0); the last row/column of tiles is truncated."""
    return [(y0, min(th, Hg - y0), x0, min(tw, Wg - x0))
            for y0 in range(0, Hg, th) for x0 in range(0, Wg, tw)]


def par_reconstruct(R, anchor_mask, wch=None, p: ParParams = ParParams(), tiles=None,
                    channels=None, with_info=False):
    """Phase-Aware Reconstruction of every skipped frame of R [F, Hg, Wg, C].

    Returns a float64 copy of R whose skipped rows are replaced by P_t(R_a, R_b)
    (Eq. block, Eq. fcpasm).  `tiles` restricts the work to a subset of tile
    indices (others are left as in R); `channels` restricts the output channels
    (the pooled sums still use every channel)."""
    R = np.asarray(R, dtype=np.float64)
    F, Hg, Wg, C = R.shape
    out = R.copy()
    assign = skipped_assignment(anchor_mask)
    all_tiles = tiles_of(Hg, Wg, p.tile_h, p.tile_w)
    sel = range(len(all_tiles)) if tiles is None else tiles
    chan = slice(None) if channels is None else np.asarray(channels)
    pairs = sorted({(a, b) for (_, a, b, _) in assign})
    info = {}
    for ti in sel:
        y0, h, x0, w = all_tiles[ti]
        bins = tile_bins(h, w)
        for (a, b) in pairs:
            Fa = rfft2_ortho(np.moveaxis(R[a, y0:y0 + h, x0:x0 + w, :], -1, 0))
            Fb = rfft2_ortho(np.moveaxis(R[b, y0:y0 + h, x0:x0 + w, :], -1, 0))
            tt = tile_transport(Fa, Fb, wch, p, bins)
            info[(ti, a, b)] = tt
            for (t, aa, bb, alpha) in assign:
                if (aa, bb) != (a, b):
                    continue
                Ft = blend(Fa[chan], Fb[chan], tt.theta, tt.g, alpha)
                rt = irfft2_ortho(Ft, w)
                out[t, y0:y0 + h, x0:x0 + w, chan] = np.moveaxis(rt, 0, -1)
    return (out, info) if with_info else out


# ===========================================================================
# Routing: pooled scores and one-block omission (Section 4.4, Eqs. pooled,
# omission; App. B.1 Eq. omissionexact), TopK initialisation (Eq. topk)
# ===========================================================================


@dataclass
class Routing:
    qbar: np.ndarray    # [K_f, H, d]
    kbar: np.ndarray    # [M, H, d]
    vbar: np.ndarray    # [M, H, d]
    s: np.ndarray       # [K_f, H, M]
    pi: np.ndarray      # [K_f, H, M]
    obar: np.ndarray    # [K_f, H, d]
    delta: np.ndarray   # [K_f, H, M, d]
    u: np.ndarray       # [K_f, H, M]


def pooled_routing(q, anchors, k_hist, v_hist, proj=None, eps=1e-8) -> Routing:
    """q [N, S, H, d]; k_hist, v_hist: the M history blocks, either an array [M, B_v, H, d]
    or a list of M arrays [n_m, H, d] (blocks of different sizes, e.g. truncated spatial
    blocks); proj: P = W_O head slices [H, d_out, d] (None: P = I).  Means over a block's
    tokens pool the statistics."""
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    qbar = np.stack([q[a].mean(axis=0) for a in anchors])          # [K_f, H, d]
    kbar = np.stack([np.asarray(b, dtype=np.float64).mean(axis=0) for b in k_hist])   # [M, H, d]
    vbar = np.stack([np.asarray(b, dtype=np.float64).mean(axis=0) for b in v_hist])
    s = np.einsum("ihd,mhd->ihm", qbar, kbar) / np.sqrt(d)          # Eq. (pooled)
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    pi = e / e.sum(axis=-1, keepdims=True)
    obar = np.einsum("ihm,mhd->ihd", pi, vbar)
    coef = pi / (1.0 - pi + eps)                                    # Eq. (omission)
    delta = coef[..., None] * (obar[:, :, None, :] - np.transpose(vbar, (1, 0, 2))[None])
    if proj is None:
        u = np.sum(delta ** 2, axis=-1)
    else:
        pd = np.einsum("hod,ihmd->ihmo", np.asarray(proj, dtype=np.float64), delta)
        u = np.sum(pd ** 2, axis=-1)
    return Routing(qbar, kbar, vbar, s, pi, obar, delta, u)


def candidate_mask(candidates, M, K=0):
    """Fixed candidate sets C_i (App. B.3): [..., M_c] distinct block indices -> boolean
    membership [..., M].  The paper requires M_c >= K_KV; a set smaller than min(K, M), a
    repeated index or one outside [0, M) raises ValueError."""
    c = np.asarray(candidates, dtype=np.int64)
    mask = np.zeros(c.shape[:-1] + (M,), dtype=bool)
    for r in np.ndindex(c.shape[:-1]):
        row = c[r]
        if np.any(row < 0) or np.any(row >= M) or len(set(row.tolist())) != len(row):
            raise ValueError("candidate indices must be distinct and inside [0, M)")
        if len(row) < min(K, M):
            raise ValueError("a candidate set smaller than the budget")
        mask[r + (row,)] = True
    return mask


def topk_blocks(score: np.ndarray, K: int, candidates=None):
    """Per (anchor, head): the K largest scores, ties to the lower block index,
    returned ascending.  K >= M or M == 0 keeps every block (routing bypass).  With
    candidate sets ([..., M_c] block indices, App. B.3) only members are eligible."""
    M = score.shape[-1]
    keff = min(K, M)
    if M == 0:
        return np.zeros(score.shape[:-1] + (0,), dtype=np.int64)
    if candidates is not None:
        score = np.where(candidate_mask(candidates, M, K), score, -np.inf)
    flat = score.reshape(-1, M)
    idx = np.empty((flat.shape[0], keff), dtype=np.int64)
    for r in range(flat.shape[0]):
        order = np.lexsort((np.arange(M), -flat[r]))               # full sort
        idx[r] = np.sort(order[:keff])
    return idx.reshape(score.shape[:-1] + (keff,))


def topk_margin(score: np.ndarray, K: int) -> np.ndarray:
    """Relative gap (s_(K) - s_(K+1)) / |s_(K)| at the selection boundary (inf if K >= M)."""
    M = score.shape[-1]
    if K >= M or K <= 0:
        return np.full(score.shape[:-1], np.inf)
    srt = -np.sort(-score, axis=-1)
    kth, nxt = srt[..., K - 1], srt[..., K]
    return (kth - nxt) / np.maximum(np.abs(kth), 1e-300)


# ===========================================================================
# Routed anchor attention (Eq. block, App. B.4): current chunk + routed blocks
# ===========================================================================


def routed_attention(q, k_cur, v_cur, k_hist, v_hist, anchors, idx, scale=None,
                     rows=None, heads=None, with_lse=False):
    """O[i, s, h, :] = sum_j softmax_j(q . k_j * scale) v_j over the current chunk
    (all N_cur * S tokens) followed by the routed history blocks idx[i, h, :] (k_hist, v_hist
    as in pooled_routing: an array of equal blocks or a list of blocks).

    Explicit max-subtracted softmax in float64.  `rows` / `heads` restrict the
    query rows / heads computed (others stay NaN)."""
    q = np.asarray(q)
    N, S, H, d = q.shape
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    Kf = len(anchors)
    rows = np.arange(S) if rows is None else np.asarray(rows)
    heads = range(H) if heads is None else heads
    O = np.full((Kf, S, H, d), np.nan)
    L = np.full((Kf, H, S), np.nan)
    kc = np.asarray(k_cur, dtype=np.float64).reshape(N * S, H, d)
    vc = np.asarray(v_cur, dtype=np.float64).reshape(N * S, H, d)
    for i, a in enumerate(anchors):
        for h in heads:
            blocks = [int(m) for m in idx[i, h]] if idx is not None else []
            keys = [kc[:, h]] + [np.asarray(k_hist[m], dtype=np.float64)[:, h] for m in blocks]
            vals = [vc[:, h]] + [np.asarray(v_hist[m], dtype=np.float64)[:, h] for m in blocks]
            kk = np.concatenate(keys)
            vv = np.concatenate(vals)
            qq = np.asarray(q[a, rows, h], dtype=np.float64)
            logits = (qq @ kk.T) * scale
            mx = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - mx)
            den = e.sum(axis=1, keepdims=True)
            O[i, rows, h] = (e / den) @ vv
            L[i, h, rows] = (mx + np.log(den))[:, 0]
    return (O, L) if with_lse else O


# ===========================================================================
# One block step at the attention residual site (Eq. block)
# ===========================================================================


def block_step(inp, K, grid, p: ParParams = ParParams(), eps=1e-8, idx=None, O=None):
    """route -> routed anchor attention -> PAR at one attention residual site.

    Returns (idx, O, r_out): r_out [N, S, H*d] holds O in the anchor rows and
    P_t(R_a, R_b) in the skipped rows (the attention output is the residual R,
    pre-W_O).  `idx` / `O` may be supplied to feed a stage the upstream result
    of another implementation (stage-by-stage parity)."""
    q = inp["q"]
    N, S, H, d = q.shape
    anchors = [int(a) for a in inp["anchors"]]
    if idx is None:
        rt = pooled_routing(q, anchors, inp["k_hist"], inp["v_hist"], eps=eps)
        idx = topk_blocks(rt.u, K)
    if O is None:
        O = routed_attention(q, inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                             anchors, idx)
    r = np.zeros((N, S, H * d))
    for i, a in enumerate(anchors):
        r[a] = np.asarray(O[i], dtype=np.float64).reshape(S, H * d)
    mask = np.zeros(N, dtype=np.uint8)
    mask[anchors] = 1
    r = par_reconstruct(r.reshape(N, grid[0], grid[1], H * d), mask, None, p)
    return idx, O, r.reshape(N, S, H * d)


# ===========================================================================
# Reconstruction-coupled routing refinement (Section 4.4, Eqs. abc, risk,
# objective, topk; App. B.2 Eqs. abcclosed, boundarycoeff, boundaryrisk;
# App. B.3 Eqs. gain, boundarygain, Alg. routing; Tab. config_cast)
# ===========================================================================


@dataclass
class RoutingCoefficients:
    """Interval coefficients of the adjacent anchor pairs (index j: anchors j-1, j) and of the
    two boundary sets (L: frames before anchor 0, pair (0, 1); R: frames after the last anchor,
    pair (J-1, J)).  Anchor positions are indices into the ordered anchor list."""
    A: np.ndarray   # [n_anchors] (entry 0 unused)
    B: np.ndarray
    C: np.ndarray
    AL: float
    BL: float
    CL: float
    AR: float
    BR: float
    CR: float


def routing_coefficients(anchors, n_frames) -> RoutingCoefficients:
    """Eq. (abc) over each interval's skipped frames and Eq. (boundarycoeff) over the boundary
    sets, with the alpha of Eq. (block)."""
    an = [int(a) for a in anchors]
    J = len(an)
    A = np.zeros(J)
    B = np.zeros(J)
    C = np.zeros(J)
    for j in range(1, J):
        a, b = an[j - 1], an[j]
        al = np.array([(t - a) / (b - a) for t in range(a + 1, b)])
        A[j] = np.sum((1 - al) ** 2)
        B[j] = np.sum(al ** 2)
        C[j] = np.sum(al * (1 - al))
    AL = BL = CL = AR = BR = CR = 0.0
    if J >= 2:
        a, b = an[0], an[1]
        al = np.array([(t - a) / (b - a) for t in range(0, a)])
        AL, BL, CL = np.sum((1 - al) ** 2), np.sum(al ** 2), np.sum(np.abs(al * (1 - al)))
        a, b = an[-2], an[-1]
        al = np.array([(t - a) / (b - a) for t in range(b + 1, n_frames)])
        AR, BR, CR = np.sum((1 - al) ** 2), np.sum(al ** 2), np.sum(np.abs(al * (1 - al)))
    return RoutingCoefficients(A, B, C, float(AL), float(BL), float(CL), float(AR), float(BR),
                               float(CR))


def _pair_risk(A, B, C, xa, xb, ua, ub):
    """Eq. (risk) summed over blocks: A (1-x_a) u_a + B (1-x_b) u_b + 2C (1-x_a)(1-x_b) sqrt(u_a u_b)."""
    return np.sum(A * (1 - xa) * ua + B * (1 - xb) * ub + 2 * C * (1 - xa) * (1 - xb) * np.sqrt(ua * ub))


def routing_objective(u, x, co: RoutingCoefficients, lam_anc=1.0, lam_rec=1.0):
    """Eq. (objective) for one head: u, x [n_anchors, M] (x binary)."""
    J = u.shape[0]
    val = lam_anc * np.sum((1 - x) * u)
    rec = 0.0
    for j in range(1, J):
        rec += _pair_risk(co.A[j], co.B[j], co.C[j], x[j - 1], x[j], u[j - 1], u[j])
    if J >= 2:   # Eq. (boundaryrisk): both sets, also when they share the pair (K_f = 2)
        rec += _pair_risk(co.AL, co.BL, co.CL, x[0], x[1], u[0], u[1])
        rec += _pair_risk(co.AR, co.BR, co.CR, x[J - 2], x[J - 1], u[J - 2], u[J - 1])
    return float(val + lam_rec * rec)


def retain_gains(i, u, x, co: RoutingCoefficients, lam_anc=1.0, lam_rec=1.0):
    """Eq. (gain) with Eq. (boundarygain): G_{i,m}, the decrease of J when anchor i keeps m."""
    J = u.shape[0]
    G = lam_anc * u[i].copy()
    if i >= 1:      # left neighbour, interval (i-1, i)
        l = i - 1
        G += lam_rec * (co.B[i] * u[i] + 2 * co.C[i] * (1 - x[l]) * np.sqrt(u[l] * u[i]))
    if i + 1 < J:   # right neighbour, interval (i, i+1)
        r = i + 1
        G += lam_rec * (co.A[r] * u[i] + 2 * co.C[r] * (1 - x[r]) * np.sqrt(u[i] * u[r]))
    if J >= 2:
        for (aq, bq, Aq, Bq, Cq) in ((0, 1, co.AL, co.BL, co.CL),
                                     (J - 2, J - 1, co.AR, co.BR, co.CR)):
            if i == aq:
                G += lam_rec * (Aq * u[i] + 2 * Cq * (1 - x[bq]) * np.sqrt(u[i] * u[bq]))
            if i == bq:
                G += lam_rec * (Bq * u[i] + 2 * Cq * (1 - x[aq]) * np.sqrt(u[i] * u[aq]))
    return G


def _mask_from_topk(score, K):
    x = np.zeros_like(score)
    if score.size:
        x[topk_blocks(score[None], K)[0]] = 1.0
    return x


def coupled_routing(u, anchors, n_frames, K, passes=2, lam_anc=1.0, lam_rec=1.0, tol=1e-6,
                    with_info=False, candidates=None):
    """Alg. (routing) for one head: u [n_anchors, M] omission scores.  Initialise every mask
    with TopK(u_i), then `passes` directional passes (forward, backward, ...) replacing M_i by
    TopK(G_i) when J drops by more than tol * max(J, 1e-8); stop after a pass with no change.
    candidates: optional fixed sets C_i ([n_anchors, M_c] block indices, App. B.3): both TopK
    run over C_i only; blocks outside C_i stay zero and still count as omissions in J and in
    the neighbours' gains.  Returns idx [n_anchors, K_eff] ascending (and the objective trace
    with with_info)."""
    u = np.asarray(u, dtype=np.float64)
    J_, M = u.shape
    keff = min(K, M)
    co = routing_coefficients(anchors, n_frames)
    cand = np.ones((J_, M), dtype=bool) if candidates is None else candidate_mask(candidates, M, K)

    def restrict(i, score):
        return np.where(cand[i], score, -np.inf)

    x = np.stack([_mask_from_topk(restrict(i, u[i]), keff) for i in range(J_)]) if M else np.zeros((J_, 0))
    trace = [routing_objective(u, x, co, lam_anc, lam_rec)]
    ambiguous = False
    if 0 < keff < M:
        for s in range(1, passes + 1):
            changed = False
            order = range(J_) if s % 2 == 1 else range(J_ - 1, -1, -1)
            for i in order:
                G = retain_gains(i, u, x, co, lam_anc, lam_rec)
                new = _mask_from_topk(restrict(i, G), keff)
                gain = float(np.sum(G * new) - np.sum(G * x[i]))
                Jcur = routing_objective(u, x, co, lam_anc, lam_rec)
                thr = tol * max(Jcur, 1e-8)
                srt = -np.sort(-G[cand[i]])
                if abs(gain - thr) <= 1e-4 * max(thr, 1e-12) or (len(srt) > keff and
                        srt[keff - 1] - srt[keff] <= 1e-4 * max(abs(srt[keff - 1]), 1e-12)):
                    ambiguous = True
                if gain > thr:
                    x[i] = new
                    changed = True
                    trace.append(routing_objective(u, x, co, lam_anc, lam_rec))
            if not changed:
                break
    idx = np.stack([np.flatnonzero(x[i]) for i in range(J_)]) if keff else np.zeros((J_, 0), int)
    if with_info:
        return idx, {"trace": trace, "ambiguous": ambiguous, "x": x, "coefficients": co}
    return idx


# ===========================================================================
# Control-aware frame selection (Section 3 "Interaction sensitivity" and "Coverage debt",
# Eqs. sensitivity, debt, score; App. B.1 Eq. normalization)
# ===========================================================================


def control_rms(delta) -> np.ndarray:
    """r_{i,k}: root mean square of the control update Delta_{i,k} over the frame's spatial and
    channel coordinates (App. B.1).  delta [N_cur, ...] -> [N_cur]."""
    d = np.asarray(delta, dtype=np.float64)
    d = d.reshape(d.shape[0], -1)
    return np.sqrt(np.mean(d * d, axis=1))


def minmax_norm(r, eps=1e-8) -> np.ndarray:
    """Eq. (normalization): (r_i - min_j r_j) / (max_j r_j - min_j r_j + eps) over the chunk."""
    r = np.asarray(r, dtype=np.float64)
    return (r - r.min()) / (r.max() - r.min() + eps)


def sensitivity(deltas, eps=1e-8):
    """Eq. (sensitivity): d_i = mean over the available control branches of Norm(Delta_{i,k});
    None when no branch supplies a fresh response."""
    if deltas is None or len(deltas) == 0:
        return None
    return np.mean([minmax_norm(control_rms(dk), eps) for dk in deltas], axis=0)


def refresh_ages(ages, anchor_mask) -> np.ndarray:
    """Eq. (debt): h^{l+1}_i = 0 for the anchors of block l, h^l_i + 1 for the other frames."""
    ages = np.asarray(ages, dtype=np.int64)
    m = np.asarray(anchor_mask).astype(bool)
    return np.where(m, 0, ages + 1)


def select_frames(deltas, ages, anchor_mask, K_f, lam_cov=0.5, eps=1e-8):
    """Eqs. (debt) and (score), then the deterministic TopK_f over all current frames with ties
    to the lower frame index.  deltas: list of the available branches' updates [N_cur, ...]
    (empty: no fresh response, the score is the debt term alone); ages, anchor_mask: [N_cur]
    refresh ages and anchors of block l.  Returns (anchors of block l+1 ascending, ages h^{l+1},
    scores S^{l+1})."""
    h = refresh_ages(ages, anchor_mask)
    N = h.shape[0]
    H_cov = -(-N // K_f)                      # ceil(N_cur / K_f)
    D = h / H_cov
    d = sensitivity(deltas, eps)
    S = lam_cov * D if d is None else d + lam_cov * D
    K = min(K_f, N)
    order = sorted(range(N), key=lambda i: (-S[i], i))
    return np.array(sorted(order[:K]), dtype=np.int64), h, S


def selection_margin(S, K_f) -> float:
    """Relative gap between the K_f-th and (K_f+1)-th largest score (inf when all frames are
    selected): a selection whose gap is tiny can flip with rounding."""
    s = np.sort(np.asarray(S, dtype=np.float64))[::-1]
    if K_f >= len(s):
        return np.inf
    return (s[K_f - 1] - s[K_f]) / max(abs(s[K_f - 1]), 1e-30)


# ===========================================================================
# Residual sites beyond the attention output (App. B.1, B.4): the output projection W_O of
# the anchor rows, and the anchor FFN whose skipped-frame residuals PAR reconstructs
# ===========================================================================


def gelu_tanh(x):
    """GELU in its tanh form, 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def linear(x, w, b=None):
    """Rows of x times w^T (+ b): x [..., D_in], w [D_out, D_in] (the layer's weight layout)."""
    y = np.asarray(x, np.float64) @ np.asarray(w, np.float64).T
    return y if b is None else y + np.asarray(b, np.float64)


def anchor_ffn(x, anchors, w1, b1, w2, b2):
    """The FFN residual of the anchor frames: GELU(x_a W1^T + b1) W2^T + b2 for every anchor
    frame a; x [F, S, D] -> [K_f, S, D]."""
    return np.stack([linear(gelu_tanh(linear(x[a], w1, b1)), w2, b2) for a in anchors])


def block_step_projected(inp, K, grid, w_o, b_o=None, p: ParParams = ParParams(), eps=1e-8,
                         idx=None, O=None):
    """Eq. (block) at the attention site with the output projection: anchor rows carry
    O_a W_O^T (+ b_O), skipped rows are PAR of those rows (App. B.1: PAR acts on the site's
    residual).  Returns (idx, O, r [N, S, D])."""
    q = inp["q"]
    N, S, H, d = q.shape
    anchors = [int(a) for a in inp["anchors"]]
    if idx is None:
        rt = pooled_routing(q, anchors, inp["k_hist"], inp["v_hist"], eps=eps)
        idx = topk_blocks(rt.u, K)
    if O is None:
        O = routed_attention(q, inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                             anchors, idx)
    r = np.zeros((N, S, H * d))
    for i, a in enumerate(anchors):
        r[a] = linear(np.asarray(O[i], np.float64).reshape(S, H * d), w_o, b_o)
    mask = np.zeros(N, dtype=np.uint8)
    mask[anchors] = 1
    r = par_reconstruct(r.reshape(N, grid[0], grid[1], H * d), mask, None, p)
    return idx, O, r.reshape(N, S, H * d)


# ===========================================================================
# Paper-granularity history blocks (App. C, Tab. config_cast: (1, 8, 8) blocks of 64
# tokens, K = ceil(0.2 M)); a block never spans frames, edge blocks are truncated
# ===========================================================================


def spatial_blocks(n_frames, Hg, Wg, bh=8, bw=8):
    """The (1, bh, bw) blocks of n_frames history frames of Hg x Wg tokens: block
    m = (f * nby + by) * nbx + bx (frame-major, then row-major over the block grid), each a
    token index array into the frame's row-major Hg * Wg tokens (rows y0..y0+h-1, columns
    x0..x0+w-1, truncated at the grid edge).  Returns [(frame, tokens), ...]."""
    nby, nbx = -(-Hg // bh), -(-Wg // bw)
    out = []
    for f in range(n_frames):
        for by in range(nby):
            for bx in range(nbx):
                ys = np.arange(by * bh, min(Hg, by * bh + bh))
                xs = np.arange(bx * bw, min(Wg, bx * bw + bw))
                out.append((f, (ys[:, None] * Wg + xs[None, :]).reshape(-1)))
    return out


def gather_blocks(frames, blocks):
    """frames [F_h, Hg * Wg, H, d] -> list of the blocks' token arrays [n_m, H, d]."""
    fr = np.asarray(frames)
    return [fr[f, tok] for f, tok in blocks]


def paper_budget(M):
    """K_KV = ceil(0.2 M) (Tab. config_cast)."""
    return int(-(-2 * M // 10))


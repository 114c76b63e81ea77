"""Plant plausible mistakes in the CPU oracle and check that its pins catch every one.

Each mutation replaces one oracle function (on the CPU, for the duration of the
test) with a subtly wrong variant: a flipped sign, a dropped term, a transposed
operand, a wrong multiplicity or tie rule.  At least one pin must then fail.
"""
import numpy as np
import pytest

import oracle.cast_oracle as O
from tests import oracle_checks as C

_orig_blend = O.blend
_orig_bins = O.tile_bins
_orig_pooled = O.pooled_routing
_orig_transport = O.tile_transport


def _blend_sign(Fa, Fb, th, g, al):
    return (1 - al) * Fa * np.exp(-1j * g * al * th) + al * Fb * np.exp(1j * g * (1 - al) * th)


def _blend_swapped(Fa, Fb, th, g, al):
    return al * Fa * np.exp(1j * g * al * th) + (1 - al) * Fb * np.exp(-1j * g * (1 - al) * th)


def _blend_no_gate(Fa, Fb, th, g, al):
    return (1 - al) * Fa * np.exp(1j * al * th) + al * Fb * np.exp(-1j * (1 - al) * th)


def _rfft2_transposed(x):
    h, w = x.shape[-2:]
    ey = O.dft_matrix(h, -1).T.conj().T        # = ey
    ex = O.dft_matrix(w, +1)[:, : w // 2 + 1]  # wrong sign of the exponent
    return (ey @ x @ ex) / np.sqrt(h * w)


def _transport_mirror_same_sign(Fa, Fb, wch, p, bins, amb_tol=1e-5):
    tt = _orig_transport(Fa, Fb, wch, p, bins, amb_tol)
    tt.theta = np.where(bins.mirror, -tt.theta, tt.theta)      # mirror copies +theta_rep
    return tt


def _transport_w_one_sided(Fa, Fb, wch, p, bins, amb_tol=1e-5):
    # Eq. (cross) with W = sum_c w_c |F_b|^2 (one anchor's power) instead of |F_b| |F_a|
    wc = np.ones(Fa.shape[0]) if wch is None else np.asarray(wch, dtype=np.float64)
    Z = np.einsum("c,cij->ij", wc, Fb * np.conj(Fa))
    W = np.einsum("c,cij->ij", wc, np.abs(Fb) ** 2)
    eta = p.eta_rel * W.max() + p.eta_abs
    Zabs = np.abs(Z)
    rel_bin = (W > eta) & (Zabs > eta)
    ry, rx = bins.rep[..., 0], bins.rep[..., 1]
    reliable = rel_bin[ry, rx]
    theta_rep = np.angle(Z[ry, rx])
    theta_rep = np.where(theta_rep <= -np.pi, np.pi, theta_rep)
    theta = np.where(bins.mirror, -theta_rep, theta_rep)
    theta = np.where(reliable & ~bins.selfconj, theta, 0.0)
    omega_plus = reliable & ~bins.dc
    if omega_plus.any():
        c = float(np.sum(bins.kappa * Zabs * omega_plus) / (np.sum(bins.kappa * W * omega_plus) + p.eps))
    else:
        c = 0.0
        theta = np.zeros_like(theta)
    tau = p.tau_low + (p.tau_high - p.tau_low) * bins.nu ** p.q
    g = 1.0 / (1.0 + np.exp(-(c - tau) / p.T))
    if p.gate_mode == "zero":
        g = np.zeros_like(g)
    elif p.gate_mode == "one":
        g = np.ones_like(g)
    if p.band_radius >= 0:
        g = np.where(bins.rho > p.band_radius, 0.0, g)
    return O.TileTransport(Z, W, eta, reliable, theta, c, g, False, False)


def _bins_kappa_one(h, w):
    b = _orig_bins(h, w)
    b.kappa = np.ones_like(b.kappa)
    return b


def _bins_nu_unnormalised(h, w):
    b = _orig_bins(h, w)
    ky = np.arange(h)[:, None]
    kx = np.arange(w // 2 + 1)[None, :]
    ky_s = np.where(ky <= (h - 1) // 2, ky, ky - h)
    b.nu = np.sqrt((ky_s / h) ** 2 + (kx / w) ** 2)
    return b


def _pooled_no_renorm(q, anchors, k, v, proj=None, eps=1e-8):
    rt = _orig_pooled(q, anchors, k, v, proj=proj, eps=eps)
    rt.delta = rt.delta * (1.0 - rt.pi[..., None] + eps)        # drops 1/(1 - pi + eps)
    rt.u = np.sum(rt.delta ** 2, axis=-1)
    return rt


def _topk_high_ties(score, K, candidates=None):
    M = score.shape[-1]
    keff = min(K, M)
    if M == 0:
        return np.zeros(score.shape[:-1] + (0,), dtype=np.int64)
    if candidates is not None:
        score = np.where(O.candidate_mask(candidates, M, K), score, -np.inf)
    flat = score.reshape(-1, M)
    out = [np.sort(np.lexsort((-np.arange(M), -r))[:keff]) for r in flat]
    return np.array(out).reshape(score.shape[:-1] + (keff,))


def _attn_ignores_history(q, kc, vc, kh, vh, anchors, idx, **kw):
    return _orig_attn(q, kc, vc, kh, vh, anchors, None if idx is None else idx[..., :0], **kw)


_orig_attn = O.routed_attention


def _attn_no_scale(q, kc, vc, kh, vh, anchors, idx, scale=None, **kw):
    return _orig_attn(q, kc, vc, kh, vh, anchors, idx, scale=1.0, **kw)


_orig_gains = O.retain_gains
_orig_coeffs = O.routing_coefficients


def _gains_no_neighbour_mask(i, u, x, co, lam_anc=1.0, lam_rec=1.0):
    return _orig_gains(i, u, np.zeros_like(x), co, lam_anc, lam_rec)   # drops the (1 - x) factor


def _gains_swapped_ab(i, u, x, co, lam_anc=1.0, lam_rec=1.0):
    sw = O.RoutingCoefficients(co.B, co.A, co.C, co.BL, co.AL, co.CL, co.BR, co.AR, co.CR)
    return _orig_gains(i, u, x, sw, lam_anc, lam_rec)


def _coeffs_signed_boundary_cross(anchors, n_frames):
    co = _orig_coeffs(anchors, n_frames)
    an = [int(a) for a in anchors]
    if len(an) >= 2:
        a, b = an[0], an[1]
        al = np.array([(t - a) / (b - a) for t in range(0, a)])
        co.CL = float(np.sum(al * (1 - al)))      # forgets |.| outside [0, 1]
    return co


_orig_norm = O.minmax_norm
_orig_sens = O.sensitivity


def _norm_from_max(r, eps=1e-8):
    r = np.asarray(r, dtype=np.float64)
    return (r.max() - r) / (r.max() - r.min() + eps)           # distance from the maximum


def _sens_absent_branch_as_zero(deltas, eps=1e-8):
    if deltas is None or len(deltas) == 0:
        return None
    n = [_orig_norm(O.control_rms(dk), eps) for dk in deltas]
    return np.sum(n, axis=0) / 2.0                              # always divides by both branches


def _ages_never_reset(ages, anchor_mask):
    return np.asarray(ages, dtype=np.int64) + 1


def _select_floor_hcov(deltas, ages, anchor_mask, K_f, lam_cov=0.5, eps=1e-8):
    h = O.refresh_ages(ages, anchor_mask)
    N = h.shape[0]
    D = h / max(N // K_f, 1)                                    # floor instead of ceil
    d = O.sensitivity(deltas, eps)
    S = lam_cov * D if d is None else d + lam_cov * D
    order = sorted(range(N), key=lambda i: (-S[i], i))
    return np.array(sorted(order[:min(K_f, N)])), h, S


def _select_ties_high(deltas, ages, anchor_mask, K_f, lam_cov=0.5, eps=1e-8):
    h = O.refresh_ages(ages, anchor_mask)
    N = h.shape[0]
    D = h / (-(-N // K_f))
    d = O.sensitivity(deltas, eps)
    S = lam_cov * D if d is None else d + lam_cov * D
    order = sorted(range(N), key=lambda i: (-S[i], -i))         # ties to the higher index
    return np.array(sorted(order[:min(K_f, N)])), h, S


def _gelu_erf(x):
    import scipy.special
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + scipy.special.erf(x / np.sqrt(2.0)))     # the erf form instead


def _linear_no_bias(x, w, b=None):
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T


def _linear_untransposed_square(x, w, b=None):
    w = np.asarray(w, np.float64)
    y = np.asarray(x, np.float64) @ (w if w.shape[0] == w.shape[1] else w.T)
    return y if b is None else y + b


_orig_spatial = O.spatial_blocks


def _spatial_blocks_padded(n_frames, Hg, Wg, bh=8, bw=8):
    # edge blocks padded to full size by repeating their first token (no partial-block mask)
    out = []
    for f, tok in _orig_spatial(n_frames, Hg, Wg, bh, bw):
        if len(tok) < bh * bw:
            tok = np.concatenate([tok, np.full(bh * bw - len(tok), tok[0])])
        out.append((f, tok))
    return out


def _budget_floor(M):
    return int(2 * M // 10)


_orig_coupled = O.coupled_routing


def _topk_candidates_ignored(score, K, candidates=None):
    return _orig_topk(score, K)


_orig_topk = O.topk_blocks


def _coupled_candidates_only_at_init(u, anchors, n_frames, K, passes=2, lam_anc=1.0, lam_rec=1.0,
                                     tol=1e-6, with_info=False, candidates=None):
    # the candidate restriction applied to the initial TopK only, not to the best responses
    if candidates is None:
        return _orig_coupled(u, anchors, n_frames, K, passes, lam_anc, lam_rec, tol, with_info)
    x0 = _orig_topk(np.asarray(u, dtype=np.float64), K, candidates=candidates)
    lifted = np.asarray(u, dtype=np.float64).copy()
    for i in range(lifted.shape[0]):
        lifted[i, x0[i]] += 1e6          # forces the same initial sets
    res = _orig_coupled(lifted, anchors, n_frames, K, passes, lam_anc, lam_rec, tol, True)
    idx, info = res
    info["x"] = np.zeros_like(lifted)
    for i in range(lifted.shape[0]):
        info["x"][i, idx[i]] = 1.0
    return (idx, info) if with_info else idx


def _coupled_noncandidates_retained(u, anchors, n_frames, K, passes=2, lam_anc=1.0, lam_rec=1.0,
                                    tol=1e-6, with_info=False, candidates=None):
    # blocks outside a neighbour's C_i treated as retained (x = 1) in the gains
    if candidates is None:
        return _orig_coupled(u, anchors, n_frames, K, passes, lam_anc, lam_rec, tol, with_info)
    cm = O.candidate_mask(candidates, np.asarray(u).shape[1])
    gains = O.retain_gains

    def patched(i, uu, x, co, la=1.0, lr=1.0):
        return gains(i, uu, np.where(cm, x, 1.0), co, la, lr)

    O.retain_gains = patched
    try:
        return _orig_coupled(u, anchors, n_frames, K, passes, lam_anc, lam_rec, tol, with_info,
                             candidates=candidates)
    finally:
        O.retain_gains = gains


MUTATIONS = {
    "candidates_ignored_in_topk": ("topk_blocks", _topk_candidates_ignored),
    "candidates_only_at_init": ("coupled_routing", _coupled_candidates_only_at_init),
    "noncandidates_retained_in_gains": ("coupled_routing", _coupled_noncandidates_retained),
    "partial_blocks_padded": ("spatial_blocks", _spatial_blocks_padded),
    "budget_floor": ("paper_budget", _budget_floor),
    "gelu_erf_form": ("gelu_tanh", _gelu_erf),
    "linear_bias_dropped": ("linear", _linear_no_bias),
    "linear_square_untransposed": ("linear", _linear_untransposed_square),
    "norm_measured_from_max": ("minmax_norm", _norm_from_max),
    "single_branch_halved": ("sensitivity", _sens_absent_branch_as_zero),
    "ages_never_reset": ("refresh_ages", _ages_never_reset),
    "coverage_scale_floor": ("select_frames", _select_floor_hcov),
    "frame_ties_high": ("select_frames", _select_ties_high),
    "gain_neighbour_mask_dropped": ("retain_gains", _gains_no_neighbour_mask),
    "gain_interval_coefficients_swapped": ("retain_gains", _gains_swapped_ab),
    "boundary_cross_without_abs": ("routing_coefficients", _coeffs_signed_boundary_cross),
    "blend_phase_sign": ("blend", _blend_sign),
    "blend_weights_swapped": ("blend", _blend_swapped),
    "blend_gate_dropped": ("blend", _blend_no_gate),
    "dft_exponent_sign": ("rfft2_ortho", _rfft2_transposed),
    "mirror_not_negated": ("tile_transport", _transport_mirror_same_sign),
    "cross_amplitude_one_sided": ("tile_transport", _transport_w_one_sided),
    "kappa_dropped": ("tile_bins", _bins_kappa_one),
    "nu_not_normalised": ("tile_bins", _bins_nu_unnormalised),
    "omission_renorm_dropped": ("pooled_routing", _pooled_no_renorm),
    "topk_ties_high": ("topk_blocks", _topk_high_ties),
    "attention_history_dropped": ("routed_attention", _attn_ignores_history),
    "attention_scale_dropped": ("routed_attention", _attn_no_scale),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, monkeypatch):
    attr, fn = MUTATIONS[name]
    monkeypatch.setattr(O, attr, fn)
    caught = []
    for check in C.ALL_CHECKS:
        try:
            check()
        except (AssertionError, ValueError, IndexError):
            caught.append(check.__name__)
    assert caught, f"no pin catches the planted mistake {name}"

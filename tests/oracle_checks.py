"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each check_* raises AssertionError on a mismatch; tests/test_oracle_pins.py runs
them on the oracle, tests/test_oracle_mutations.py plants plausible mistakes in
the oracle and asserts that some check catches each one.  Nothing here calls the
CUDA path.
"""
from __future__ import annotations

import itertools
import math
import os

import numpy as np
import scipy.special

import oracle.cast_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


# ---------------------------------------------------------------------------
# DFT (Section 4.3, App. A.2)
# ---------------------------------------------------------------------------


def check_dft_matches_library():
    """The naive DFT equals numpy's orthonormal rfft2 for every tile shape up to 8x8."""
    r = _rng(0)
    for h in range(1, 9):
        for w in range(1, 9):
            x = r.standard_normal((3, h, w))
            assert np.allclose(O.rfft2_ortho(x), np.fft.rfft2(x, norm="ortho"), atol=1e-12)


def check_dft_round_trip_and_parseval():
    """irfft2(rfft2(x)) = x and sum kappa |F|^2 = sum x^2 (real-FFT multiplicities)."""
    r = _rng(1)
    for h, w in [(8, 8), (4, 8), (8, 4), (6, 8), (5, 7), (3, 3), (1, 8), (8, 1), (2, 2)]:
        x = r.standard_normal((4, h, w))
        F = O.rfft2_ortho(x)
        assert np.allclose(O.irfft2_ortho(F, w), x, atol=1e-12)
        b = O.tile_bins(h, w)
        assert np.allclose(np.sum(b.kappa * np.abs(F) ** 2, axis=(-2, -1)),
                           np.sum(x ** 2, axis=(-2, -1)), rtol=1e-12)


def check_bin_structure():
    """Mirrors hold the conjugate of their representative for real input; self-conjugate
    bins are real; every stored bin's (ky, kx) radius is within [0, 1] after normalisation."""
    r = _rng(2)
    for h in range(1, 9):
        for w in range(1, 9):
            x = r.standard_normal((h, w))
            F = np.fft.rfft2(x, norm="ortho")
            b = O.tile_bins(h, w)
            ry, rx = b.rep[..., 0], b.rep[..., 1]
            assert np.allclose(F[b.mirror], np.conj(F[ry, rx][b.mirror]), atol=1e-12)
            assert np.allclose(F[b.selfconj].imag, 0.0, atol=1e-12)
            assert b.nu.min() >= 0.0 and b.nu.max() <= 1.0 + 1e-15
            if h % 2 == 0 and w % 2 == 0:
                assert b.selfconj.sum() == 4
                assert abs(b.nu[h // 2, w // 2] - 1.0) < 1e-15


# ---------------------------------------------------------------------------
# PAR (Section 4.3, Eq. fcpasm; App. A.2)
# ---------------------------------------------------------------------------


def _assign(mask):
    return O.skipped_assignment(mask)


def check_interval_coefficients_closed_form():
    """Sums of (1-a)^2, a^2, a(1-a) over an interval's skipped frames (Eq. abc) with the
    alphas of Eq. (block) equal the printed closed forms of Eq. (abcclosed)."""
    for n, A_ref, C_ref in read_golden("abc_closed_form.txt"):
        n = int(n)
        mask = np.zeros(n + 1, dtype=np.uint8)
        mask[0] = mask[n] = 1
        al = np.array([a for (_, _, _, a) in _assign(mask)]) if n > 1 else np.zeros(0)
        assert abs(np.sum((1 - al) ** 2) - float(A_ref)) < 1e-12
        assert abs(np.sum(al ** 2) - float(A_ref)) < 1e-12
        assert abs(np.sum(al * (1 - al)) - float(C_ref)) < 1e-12


def check_assignment_boundaries():
    """Frames outside the anchor span extrapolate from the two nearest anchors (Eq. block)."""
    got = {t: (a, b, al) for (t, a, b, al) in _assign([0, 1, 0, 1, 0, 0])}
    assert got[0] == (1, 3, -0.5)
    assert got[2] == (1, 3, 0.5)
    assert got[4] == (1, 3, 1.5) and got[5] == (1, 3, 2.0)
    assert _assign([1, 1, 1]) == []


def _par(R, mask, **kw):
    wch = kw.pop("wch", None)
    return O.par_reconstruct(R, np.asarray(mask, dtype=np.uint8), wch, O.ParParams(**kw))


def check_par_identical_anchors():
    """R_a = R_b: theta = 0, every reconstruction returns the anchor (interpolation and
    extrapolation, every gate mode, ragged edge tiles)."""
    r = _rng(3)
    base = r.standard_normal((11, 13, 5))
    R = np.stack([base] * 6)
    R[[1, 2, 4, 5]] = r.standard_normal((4, 11, 13, 5))   # skipped rows: overwritten
    for mode in ("paper", "zero", "one"):
        out = _par(R, [1, 0, 0, 1, 0, 0], gate_mode=mode)
        for t in (1, 2, 4, 5):
            assert np.allclose(out[t], base, atol=1e-12)


def check_par_gate_zero_is_linear():
    """g = 0 gives direct value interpolation / extrapolation (1-a) R_a + a R_b."""
    r = _rng(4)
    R = r.standard_normal((7, 10, 12, 6))
    mask = [0, 1, 0, 0, 1, 0, 0]
    out = _par(R, mask, gate_mode="zero")
    for (t, a, b, al) in _assign(mask):
        assert np.allclose(out[t], (1 - al) * R[a] + al * R[b], atol=1e-12)
    for (t, a, b, al) in _assign(mask):   # band radius 0 keeps only DC -> also linear
        out2 = _par(R, mask, band_radius=0.0)
        assert np.allclose(out2[t], (1 - al) * R[a] + al * R[b], atol=1e-12)


def check_par_endpoints():
    """alpha = 0 reproduces R_a and alpha = 1 reproduces R_b exactly (Section 4.3)."""
    r = _rng(5)
    F_a = O.rfft2_ortho(r.standard_normal((3, 8, 8)))
    F_b = O.rfft2_ortho(r.standard_normal((3, 8, 8)))
    th = r.uniform(-np.pi, np.pi, (8, 5))
    g = r.uniform(0, 1, (8, 5))
    assert np.allclose(O.blend(F_a, F_b, th, g, 0.0), F_a, atol=1e-14)
    assert np.allclose(O.blend(F_a, F_b, th, g, 1.0), F_b, atol=1e-14)


def _bandlimited_tile(r, C, h, w, keep):
    """Real [C, h, w] fields whose spectrum lives on the bins where keep(ky_s, kx) holds."""
    F = np.fft.rfft2(r.standard_normal((C, h, w)), norm="ortho")
    ky = np.fft.fftfreq(h, 1.0 / h)[:, None]
    kx = np.arange(w // 2 + 1)[None, :]
    F = F * keep(ky, kx)
    return np.fft.irfft2(F, s=(h, w), norm="ortho")


def check_par_translation_identity():
    """Eq. (exacttranslation): with g = 1, a band-limited circular translation by d between
    the anchors reconstructs to the translation by alpha*d, also for alpha outside [0, 1]."""
    r = _rng(6)
    # shift along W by 2: energy only at |kx| <= 1 so that |omega . d| < pi
    x = _bandlimited_tile(r, 3, 8, 8, lambda ky, kx: (kx <= 1))
    R = np.zeros((5, 8, 8, 3))
    R[0] = np.moveaxis(x, 0, -1)
    R[2] = np.roll(R[0], 2, axis=1)
    out = _par(R, [1, 0, 1, 0, 0], gate_mode="one")
    assert np.allclose(out[1], np.roll(R[0], 1, axis=1), atol=1e-10)      # alpha = 1/2
    assert np.allclose(out[4], np.roll(R[0], 4, axis=1), atol=1e-10)      # alpha = 2
    # shift along H by 2 (tests the mirrored kx = 0 column): energy at |ky| <= 1
    y = _bandlimited_tile(r, 3, 8, 8, lambda ky, kx: (np.abs(ky) <= 1) + 0 * kx)
    R = np.zeros((4, 8, 8, 3))
    R[1] = np.moveaxis(y, 0, -1)
    R[3] = np.roll(R[1], 2, axis=0)
    out = _par(R, [0, 1, 0, 1], gate_mode="one")
    assert np.allclose(out[2], np.roll(R[1], 1, axis=0), atol=1e-10)      # alpha = 1/2
    assert np.allclose(out[0], np.roll(R[1], -1, axis=0), atol=1e-10)     # alpha = -1/2
    # diagonal shift (1, 1) with energy in the low band: alpha = 3 extrapolates by (3, 3)
    z = _bandlimited_tile(r, 2, 8, 8, lambda ky, kx: (np.abs(ky) <= 1) & (kx <= 1))
    R = np.zeros((5, 8, 8, 2))
    R[0] = np.moveaxis(z, 0, -1)
    R[1] = np.roll(R[0], (1, 1), axis=(0, 1))
    out = _par(R, [1, 1, 0, 0, 0], gate_mode="one")
    assert np.allclose(out[3], np.roll(R[0], (3, 3), axis=(0, 1)), atol=1e-10)


def check_par_confidence_closed_form():
    """Two channels carrying one spatial frequency, translated by d1 and d2: the pooled
    resultant length gives c = |cos(omega.(d1 - d2)/2)|; a pure translation gives c = 1."""
    h = w = 8
    yy, xx = np.meshgrid(np.arange(h), np.arange(w), indexing="ij")
    k = (0, 1)                      # one bin pair
    om = 2 * np.pi * np.array([k[0] / h, k[1] / w])
    base = np.cos(om[0] * yy + om[1] * xx + 0.3)
    for d1, d2 in [((0, 1), (0, 1)), ((0, 1), (0, 3)), ((0, 0), (0, 2)), ((0, 2), (0, 3))]:
        A = np.stack([base, base])
        B = np.stack([np.roll(base, d1, axis=(0, 1)), np.roll(base, d2, axis=(0, 1))])
        Fa, Fb = O.rfft2_ortho(A), O.rfft2_ortho(B)
        tt = O.tile_transport(Fa, Fb, None, O.ParParams(), O.tile_bins(h, w))
        delta = om @ (np.array(d1) - np.array(d2))
        assert abs(tt.c - abs(np.cos(delta / 2))) < 1e-9, (d1, d2, tt.c)
    # content at (1, 0) (kappa = 1, stored with its mirror) and at (0, 1) (kappa = 2) with
    # coherence 1 and |cos(pi/4)|: c weighs every bin of the full spectrum equally
    om1, om2 = 2 * np.pi / h, 2 * np.pi / w
    f1 = np.cos(om1 * yy + 0.2)
    f2 = np.cos(om2 * xx + 0.7)
    A = np.stack([f1 + f2, f1 + f2])
    B = np.stack([np.roll(f1, 1, axis=0) + np.roll(f2, 1, axis=1),
                  np.roll(f1, 1, axis=0) + np.roll(f2, 3, axis=1)])
    tt = O.tile_transport(O.rfft2_ortho(A), O.rfft2_ortho(B), None, O.ParParams(),
                          O.tile_bins(h, w))
    assert abs(tt.c - (1.0 + abs(np.cos(np.pi / 4))) / 2.0) < 1e-9, tt.c
    # random content with independent random circular shifts per channel: 0 <= c <= 1
    r = _rng(7)
    A = r.standard_normal((64, 8, 8))
    B = np.stack([np.roll(a, tuple(r.integers(0, 8, 2)), axis=(0, 1)) for a in A])
    tt = O.tile_transport(O.rfft2_ortho(A), O.rfft2_ortho(B), None, O.ParParams(),
                          O.tile_bins(8, 8))
    assert 0.0 <= tt.c <= 0.6


def check_par_gate_at_threshold():
    """Eq. (gate): where c equals tau(nu) the gate is exactly 1/2; the printed constants
    (tau_low, tau_high, q, T) of Tab. config_cast fix tau at nu = 0 and nu = 1."""
    consts = {k: float(v) for k, v in read_golden("par_constants.txt")}
    p = O.ParParams()
    for k in ("tau_low", "tau_high", "q", "T", "eta_rel", "eta_abs", "eps"):
        assert getattr(p, k) == consts[k], k
    assert (p.tile_h, p.tile_w) == (int(consts["tile_h"]), int(consts["tile_w"]))
    h = w = 8
    b = O.tile_bins(h, w)
    yy, xx = np.meshgrid(np.arange(h), np.arange(w), indexing="ij")
    # bin (0, 1): nu = (1/8) / sqrt(0.5); tau = 0.25 + 0.5 nu^2 = 0.265625
    nu = b.nu[0, 1]
    tau = consts["tau_low"] + (consts["tau_high"] - consts["tau_low"]) * nu ** consts["q"]
    assert abs(tau - 0.265625) < 1e-15
    # two channels at frequency (0,1) with translations differing by delta along W give
    # c = |cos(delta * pi / 8)|; pick delta so that c = tau
    delta = 8.0 / np.pi * np.arccos(tau)
    om = 2 * np.pi / w
    base = np.cos(om * xx + 0.1)
    A = np.stack([base, base])
    B = np.stack([np.cos(om * (xx - 0.0) + 0.1), np.cos(om * (xx - delta) + 0.1)])
    tt = O.tile_transport(O.rfft2_ortho(A), O.rfft2_ortho(B), None, p, b)
    assert abs(tt.c - tau) < 1e-9
    assert abs(tt.g[0, 1] - 0.5) < 1e-7


def check_par_frozen_transport_bound():
    """Prop. 1 (Eq. bound) and the extrapolation amplification bound |1-a| + |a| (App. A.2):
    with U and g frozen, perturbations of the anchors move the reconstruction by at most
    the stated amounts."""
    r = _rng(8)
    h = w = 8
    b = O.tile_bins(h, w)
    Ra, Rb = r.standard_normal((2, 4, h, w))
    tt = O.tile_transport(O.rfft2_ortho(Ra), O.rfft2_ortho(Rb), None, O.ParParams(), b)
    for n in (2, 3, 5):
        alphas = np.arange(1, n) / n
        va, vb = r.standard_normal((2, 4, h, w))
        Fa, Fb = O.rfft2_ortho(va), O.rfft2_ortho(vb)
        lhs = sum(np.sum(O.irfft2_ortho(O.blend(Fa, Fb, tt.theta, tt.g, al), w) ** 2)
                  for al in alphas)
        A = np.sum((1 - alphas) ** 2)
        B = np.sum(alphas ** 2)
        C = np.sum(alphas * (1 - alphas))
        na, nb = np.linalg.norm(va), np.linalg.norm(vb)
        assert lhs <= A * na ** 2 + B * nb ** 2 + 2 * C * na * nb + 1e-9
        # frozen transport is norm preserving per anchor (Parseval)
        one_a = O.irfft2_ortho(O.blend(Fa, 0 * Fb, tt.theta, tt.g, 0.5), w) / 0.5
        assert abs(np.linalg.norm(one_a) - na) < 1e-9
    for al in (-1.0, -0.5, 1.5, 2.0):
        va, vb = r.standard_normal((2, 4, h, w))
        out = O.irfft2_ortho(O.blend(O.rfft2_ortho(va), O.rfft2_ortho(vb), tt.theta, tt.g, al), w)
        assert np.linalg.norm(out) <= (abs(1 - al) + abs(al)) * max(
            np.linalg.norm(va), np.linalg.norm(vb)) + 1e-9


def check_par_unreliable_bins_interpolate():
    """A bin with no energy in one anchor fails the reliability threshold and keeps U = 1."""
    h = w = 8
    r = _rng(9)
    A = _bandlimited_tile(r, 2, h, w, lambda ky, kx: (kx <= 2))
    B = _bandlimited_tile(r, 2, h, w, lambda ky, kx: (kx <= 1))     # kx = 2 empty in B
    tt = O.tile_transport(O.rfft2_ortho(A), O.rfft2_ortho(B), None, O.ParParams(),
                          O.tile_bins(h, w))
    assert not tt.reliable[:, 2].any()
    assert np.all(tt.theta[:, 2] == 0.0)
    assert not tt.reliable[0, 0] or tt.theta[0, 0] == 0.0


def check_par_weights_scale_invariant():
    """Scaling every channel weight by a constant leaves the reconstruction unchanged;
    unit weights equal the unweighted paper form."""
    r = _rng(10)
    R = r.standard_normal((3, 8, 16, 6))
    mask = [1, 0, 1]
    wc = r.uniform(0.1, 1.0, 6)
    a = _par(R, mask, wch=wc)
    b = _par(R, mask, wch=3.0 * wc)
    c = _par(R, mask, wch=np.ones(6))
    d = _par(R, mask)
    assert np.allclose(a, b, atol=1e-9)
    assert np.allclose(c, d, atol=1e-12)


def check_par_time_reversal():
    """Reversing the frames swaps the two anchors of every pair and maps alpha to 1 - alpha
    (Eq. block); the pooled Z becomes conj(Z) while W, c and g stay the same (Eqs. cross,
    confidence, gate), and Eq. (fcpasm) with theta -> -theta then reconstructs the same frames.
    So PAR of the reversed sequence, reversed back, equals PAR of the sequence: the paper's
    gate on non-translating fields, interpolated and extrapolated frames, ragged edge tiles and
    channel weights."""
    r = _rng(32)
    R = r.standard_normal((9, 11, 13, 6))
    mask = [0, 1, 0, 0, 1, 0, 1, 0, 0]
    wc = r.uniform(0.5, 2.0, 6)
    fwd, info = O.par_reconstruct(R, np.asarray(mask, dtype=np.uint8), wc, O.ParParams(),
                                  with_info=True)
    assert not any(tt.branch_ambiguous for tt in info.values())   # theta away from +-pi
    rev = _par(R[::-1].copy(), mask[::-1], wch=wc)[::-1]
    assert np.allclose(fwd, rev, atol=1e-10)


# ---------------------------------------------------------------------------
# Routing (Section 4.4, Eqs. pooled, omission; App. B.1 Eq. omissionexact)
# ---------------------------------------------------------------------------


def _routing_inputs(seed, N=3, S=5, H=2, d=4, M=6, Bv=3):
    r = _rng(seed)
    q = r.standard_normal((N, S, H, d)) + r.standard_normal((N, 1, H, d))
    k = r.standard_normal((M, Bv, H, d)) + r.standard_normal((M, 1, H, d))
    v = r.standard_normal((M, Bv, H, d)) + r.standard_normal((M, 1, H, d))
    return q, k, v


def check_omission_identity():
    """Eq. (omissionexact): with eps = 0, delta_m equals the change of the pooled output when
    block m is dropped and the remaining weights are renormalised (brute force)."""
    q, k, v = _routing_inputs(11)
    anchors = [0, 2]
    rt = O.pooled_routing(q, anchors, k, v, eps=0.0)
    M, H, d = k.shape[0], k.shape[2], k.shape[3]
    for i, a in enumerate(anchors):
        for h in range(H):
            qb = q[a, :, h].mean(axis=0)
            kb = k[:, :, h].mean(axis=1)
            vb = v[:, :, h].mean(axis=1)
            s = kb @ qb / np.sqrt(d)
            full = scipy.special.softmax(s) @ vb
            assert np.allclose(rt.obar[i, h], full, atol=1e-12)
            for m in range(M):
                keep = [j for j in range(M) if j != m]
                drop = scipy.special.softmax(s[keep]) @ vb[keep]
                assert np.allclose(rt.delta[i, h, m], drop - full, atol=1e-10)


def check_omission_projection():
    """u = ||P delta||^2: P = I gives ||delta||^2, an orthogonal P leaves u unchanged, P = 2I
    multiplies it by 4, and u equals delta^T (P^T P) delta (the Gram form)."""
    q, k, v = _routing_inputs(12)
    H, d = q.shape[2], q.shape[3]
    r = _rng(13)
    base = O.pooled_routing(q, [1], k, v)
    Qm = np.stack([np.linalg.qr(r.standard_normal((d, d)))[0] for _ in range(H)])
    rot = O.pooled_routing(q, [1], k, v, proj=Qm)
    two = O.pooled_routing(q, [1], k, v, proj=2 * np.stack([np.eye(d)] * H))
    assert np.allclose(base.u, np.sum(base.delta ** 2, axis=-1), rtol=1e-12)
    assert np.allclose(rot.u, base.u, rtol=1e-10)
    assert np.allclose(two.u, 4 * base.u, rtol=1e-12)
    P = r.standard_normal((H, 7, d))
    pr = O.pooled_routing(q, [1], k, v, proj=P)
    gram = np.einsum("hod,hoe->hde", P, P)
    assert np.allclose(pr.u, np.einsum("ihmd,hde,ihme->ihm", pr.delta, gram, pr.delta),
                       rtol=1e-10)


def check_pooled_scores():
    """s = q.k/sqrt(d) on token means, softmax over blocks sums to one, scores permute with
    the blocks (Eq. pooled)."""
    q, k, v = _routing_inputs(14)
    rt = O.pooled_routing(q, [0, 1], k, v)
    d = q.shape[-1]
    assert np.allclose(rt.pi.sum(-1), 1.0)
    for i, a in enumerate([0, 1]):
        for h in range(q.shape[2]):
            for m in range(k.shape[0]):
                qs = sum(q[a, s, h] for s in range(q.shape[1])) / q.shape[1]
                ks = sum(k[m, j, h] for j in range(k.shape[1])) / k.shape[1]
                assert abs(rt.s[i, h, m] - float(qs @ ks) / np.sqrt(d)) < 1e-12
    perm = _rng(15).permutation(k.shape[0])
    rp = O.pooled_routing(q, [0, 1], k[perm], v[perm])
    assert np.allclose(rp.u, rt.u[..., perm], rtol=1e-12)


def check_topk():
    """TopK keeps the K largest (the subset of maximal sum when scores are distinct), ties
    go to the lower block index, output ascending; K >= M keeps every block."""
    r = _rng(16)
    for _ in range(20):
        M, K = 7, 3
        u = r.standard_normal(M)
        best = max(itertools.combinations(range(M), K), key=lambda c: sum(u[list(c)]))
        assert list(O.topk_blocks(u[None], K)[0]) == sorted(best)
    u = np.array([1.0, 3.0, 2.0, 3.0, 2.0, 0.5])
    assert list(O.topk_blocks(u[None], 3)[0]) == [1, 2, 3]
    assert list(O.topk_blocks(u[None], 2)[0]) == [1, 3]
    assert list(O.topk_blocks(u[None], 9)[0]) == list(range(6))
    assert O.topk_blocks(np.zeros((1, 0)), 3).shape == (1, 0)


# ---------------------------------------------------------------------------
# Routed attention (Eq. block; App. B.4)
# ---------------------------------------------------------------------------


def _attn_inputs(seed, N=3, S=4, H=2, d=8, M=3, Bv=5):
    r = _rng(seed)
    return (r.standard_normal((N, S, H, d)), r.standard_normal((N, S, H, d)),
            r.standard_normal((N, S, H, d)), r.standard_normal((M, Bv, H, d)),
            r.standard_normal((M, Bv, H, d)))


def check_attention_brute_force():
    """Pure-Python loops of softmax attention over the current chunk followed by the routed
    blocks equal the oracle on tiny inputs."""
    q, kc, vc, kh, vh = _attn_inputs(17)
    N, S, H, d = q.shape
    anchors = [0, 2]
    idx = np.array([[[0, 2], [1, 2]], [[1, 2], [0, 1]]])
    out = O.routed_attention(q, kc, vc, kh, vh, anchors, idx)
    sc = 1 / np.sqrt(d)
    for i, a in enumerate(anchors):
        for h in range(H):
            keys = [kc[f, s, h] for f in range(N) for s in range(S)]
            vals = [vc[f, s, h] for f in range(N) for s in range(S)]
            for m in idx[i, h]:
                keys += [kh[m, j, h] for j in range(kh.shape[1])]
                vals += [vh[m, j, h] for j in range(kh.shape[1])]
            for s in range(S):
                lg = [float(q[a, s, h] @ kk) * sc for kk in keys]
                mx = max(lg)
                e = [np.exp(x - mx) for x in lg]
                z = sum(e)
                o = sum(ej / z * vv for ej, vv in zip(e, vals))
                assert np.allclose(out[i, s, h], o, atol=1e-12)


def check_attention_dense_limit():
    """Routing every history block equals dense softmax attention over current plus all
    history (library softmax), and permuting the routed blocks changes nothing."""
    q, kc, vc, kh, vh = _attn_inputs(18)
    N, S, H, d = q.shape
    M = kh.shape[0]
    anchors = [1]
    idx = np.tile(np.arange(M), (1, H, 1))
    out = O.routed_attention(q, kc, vc, kh, vh, anchors, idx)
    for h in range(H):
        K = np.concatenate([kc[:, :, h].reshape(-1, d), kh[:, :, h].reshape(-1, d)])
        V = np.concatenate([vc[:, :, h].reshape(-1, d), vh[:, :, h].reshape(-1, d)])
        ref = scipy.special.softmax(q[1, :, h] @ K.T / np.sqrt(d), axis=1) @ V
        assert np.allclose(out[0, :, h], ref, atol=1e-12)
    perm = idx[..., ::-1]
    assert np.allclose(O.routed_attention(q, kc, vc, kh, vh, anchors, perm), out, atol=1e-12)


# ---------------------------------------------------------------------------
# Coupled routing refinement (Section 4.4 Eqs. abc, risk, objective, topk; App. B.2, B.3)
# ---------------------------------------------------------------------------


def check_routing_coefficients():
    """Interior coefficients equal the closed forms of Eq. (abcclosed); boundary coefficients make
    the frozen-transport extrapolation bound (App. B.2) hold and be attained: with U and g frozen,
    sum over the boundary frames of ||(1-a) T_a v_a + a T_b v_b||^2 is at most
    A_q |v_a|^2 + B_q |v_b|^2 + 2 C_q |v_a| |v_b|, with equality for g = 0 and v_b = -v_a."""
    for n, A_ref, C_ref in read_golden("abc_closed_form.txt"):
        co = O.routing_coefficients([2, 2 + int(n)], 4 + int(n))
        assert abs(co.A[1] - float(A_ref)) < 1e-12 and abs(co.B[1] - float(A_ref)) < 1e-12
        assert abs(co.C[1] - float(C_ref)) < 1e-12
    r = _rng(20)
    h = w = 8
    b = O.tile_bins(h, w)
    Ra, Rb = r.standard_normal((2, 3, h, w))
    tt = O.tile_transport(O.rfft2_ortho(Ra), O.rfft2_ortho(Rb), None, O.ParParams(), b)
    anchors, F = [3, 5, 6], 10          # left set {0,1,2} with pair (3,5); right set {7,8,9} with (5,6)
    co = O.routing_coefficients(anchors, F)
    for (a, bb, Aq, Bq, Cq, frames) in ((3, 5, co.AL, co.BL, co.CL, range(0, 3)),
                                        (5, 6, co.AR, co.BR, co.CR, range(7, 10))):
        va = r.standard_normal((3, h, w))
        vb = r.standard_normal((3, h, w))
        Fa, Fb = O.rfft2_ortho(va), O.rfft2_ortho(vb)
        lhs = sum(np.sum(O.irfft2_ortho(O.blend(Fa, Fb, tt.theta, tt.g, (t - a) / (bb - a)), w) ** 2)
                  for t in frames)
        na, nb = np.linalg.norm(va), np.linalg.norm(vb)
        assert lhs <= Aq * na ** 2 + Bq * nb ** 2 + 2 * Cq * na * nb + 1e-9
        z = np.zeros_like(tt.g)
        eq = sum(np.sum(O.irfft2_ortho(O.blend(Fa, -Fa, tt.theta, z, (t - a) / (bb - a)), w) ** 2)
                 for t in frames)
        assert abs(eq - (Aq + Bq + 2 * Cq) * na ** 2) < 1e-9 * max(1.0, eq)


def check_retain_gain_linearity():
    """Holding the other masks fixed, J = constant - sum_m x_{i,m} G_{i,m} (App. B.3): flipping
    x_{i,m} changes Eq. (objective) by exactly -G_{i,m}, for interior and boundary anchors,
    including K_f = 2 where both boundary sets share the pair."""
    r = _rng(21)
    for anchors, F, M in (([1, 3, 4, 8], 11, 5), ([2, 5], 9, 4), ([0, 2, 4, 6], 8, 3)):
        J = len(anchors)
        u = r.exponential(size=(J, M))
        x = (r.uniform(size=(J, M)) < 0.5).astype(float)
        co = O.routing_coefficients(anchors, F)
        lam = (0.7, 1.3)
        for i in range(J):
            G = O.retain_gains(i, u, x, co, *lam)
            for m in range(M):
                x1, x0 = x.copy(), x.copy()
                x1[i, m], x0[i, m] = 1.0, 0.0
                d = O.routing_objective(u, x1, co, *lam) - O.routing_objective(u, x0, co, *lam)
                assert abs(d + G[m]) < 1e-9 * max(1.0, abs(G[m])), (anchors, i, m)


def check_coupled_routing():
    """Alg. (routing): every anchor keeps exactly K blocks, J never increases, the result is no
    worse than independent TopK, lambda_rec = 0 gives independent TopK, and once passes stop
    changing, no single anchor can lower J with any K-subset (brute force)."""
    r = _rng(22)
    for trial in range(12):
        anchors = sorted(r.choice(9, size=int(r.integers(2, 5)), replace=False).tolist())
        M, K = 6, 2
        u = r.exponential(size=(len(anchors), M)) * r.uniform(0.2, 3.0, size=(1, M))
        idx, info = O.coupled_routing(u, anchors, 9, K, passes=2, with_info=True)
        assert idx.shape == (len(anchors), K)
        assert all(len(set(row)) == K for row in idx)
        tr = info["trace"]
        assert all(b <= a + 1e-12 for a, b in zip(tr, tr[1:]))
        co = O.routing_coefficients(anchors, 9)
        xi = np.zeros_like(u)
        ind = O.topk_blocks(u, K)
        for i in range(len(anchors)):
            xi[i, ind[i]] = 1
        assert O.routing_objective(u, info["x"], co) <= O.routing_objective(u, xi, co) + 1e-12
        assert np.array_equal(O.coupled_routing(u, anchors, 9, K, lam_rec=0.0), ind)
        idx50, info50 = O.coupled_routing(u, anchors, 9, K, passes=60, with_info=True)
        x = info50["x"]
        J0 = O.routing_objective(u, x, co)
        for i in range(len(anchors)):
            for sub in itertools.combinations(range(M), K):
                y = x.copy()
                y[i] = 0
                y[i, list(sub)] = 1
                assert O.routing_objective(u, y, co) >= J0 - 1e-6 * max(J0, 1e-8) - 1e-12
    u = r.exponential(size=(3, 4))
    assert np.array_equal(O.coupled_routing(u, [0, 2, 4], 5, 7), np.tile(np.arange(4), (3, 1)))



def _random_candidates(r, J, M, Mc):
    return np.stack([np.sort(r.choice(M, size=Mc, replace=False)) for _ in range(J)])


def check_candidate_topk():
    """Fixed candidate sets (App. B.3): TopK runs over C_i only (the K-subset of C_i with the
    largest sum, brute force), C_i = all blocks is the unrestricted TopK, and a set smaller than
    the budget or with a repeated / out-of-range index is rejected."""
    r = _rng(23)
    for _ in range(20):
        M, K, Mc = 8, 3, 5
        u = r.standard_normal((2, M))
        c = _random_candidates(r, 2, M, Mc)
        got = O.topk_blocks(u, K, candidates=c)
        for i in range(2):
            best = max(itertools.combinations(c[i].tolist(), K), key=lambda t: sum(u[i, list(t)]))
            assert list(got[i]) == sorted(best)
        assert np.array_equal(O.topk_blocks(u, K, candidates=np.tile(np.arange(M), (2, 1))),
                              O.topk_blocks(u, K))
    for bad in ([[0, 1]], [[0, 0, 1]], [[0, 1, 9]]):
        try:
            O.topk_blocks(np.zeros((1, 8)), 3, candidates=np.array(bad))
        except ValueError:
            continue
        raise AssertionError(f"candidate set {bad} accepted")


def check_candidate_coupled_routing():
    """Alg. (routing) with fixed candidate sets: every kept block lies in C_i, J never
    increases, the result is no worse than independent TopK over the same sets, C_i = all
    blocks reproduces the unrestricted refinement, and at a fixed point no anchor can lower J
    (blocks outside C_i counted as omitted) with any K-subset of its own C_i (brute force)."""
    r = _rng(24)
    for trial in range(12):
        anchors = sorted(r.choice(9, size=int(r.integers(2, 5)), replace=False).tolist())
        J, M, K, Mc = len(anchors), 7, 2, 4
        u = r.exponential(size=(J, M)) * r.uniform(0.2, 3.0, size=(1, M))
        c = _random_candidates(r, J, M, Mc)
        cm = O.candidate_mask(c, M)
        co = O.routing_coefficients(anchors, 9)
        idx, info = O.coupled_routing(u, anchors, 9, K, passes=60, with_info=True, candidates=c)
        assert idx.shape == (J, K)
        assert all(cm[i, idx[i]].all() for i in range(J))
        tr = info["trace"]
        assert all(b <= a + 1e-12 for a, b in zip(tr, tr[1:]))
        ind = O.topk_blocks(u, K, candidates=c)
        xi = np.zeros_like(u)
        for i in range(J):
            xi[i, ind[i]] = 1
        x = info["x"]
        J0 = O.routing_objective(u, x, co)
        assert J0 <= O.routing_objective(u, xi, co) + 1e-12
        for i in range(J):
            for sub in itertools.combinations(c[i].tolist(), K):
                y = x.copy()
                y[i] = 0
                y[i, list(sub)] = 1
                assert O.routing_objective(u, y, co) >= J0 - 1e-6 * max(J0, 1e-8) - 1e-12
        full = np.tile(np.arange(M), (J, 1))
        assert np.array_equal(O.coupled_routing(u, anchors, 9, K, candidates=full),
                              O.coupled_routing(u, anchors, 9, K))


# ----------------------------------------------------------------------------------------------
# Control-aware frame selection (Eqs. sensitivity, normalization, debt, score)
# ----------------------------------------------------------------------------------------------

def check_control_rms_brute_force():
    """r_{i,k} against pure-Python loops over every coordinate of each frame (App. B.1)."""
    rng = np.random.default_rng(11)
    delta = rng.standard_normal((3, 4, 5, 2))
    r = O.control_rms(delta)
    for i in range(3):
        acc, n = 0.0, 0
        for a in range(4):
            for b in range(5):
                for c in range(2):
                    acc += float(delta[i, a, b, c]) ** 2
                    n += 1
        assert abs(r[i] - math.sqrt(acc / n)) < 1e-12


def check_minmax_normalization():
    """Eq. (normalization): closed forms, a constant response contributes zero, range [0, 1)."""
    got = O.minmax_norm([1.0, 2.0, 3.0], eps=0.0)
    assert np.allclose(got, [0.0, 0.5, 1.0])
    got = O.minmax_norm([5.0, 1.0, 3.0], eps=1e-8)
    assert np.allclose(got, [4.0 / (4.0 + 1e-8), 0.0, 2.0 / (4.0 + 1e-8)], rtol=0, atol=1e-15)
    assert np.all(O.minmax_norm([2.5, 2.5, 2.5]) == 0.0)
    rng = np.random.default_rng(3)
    v = O.minmax_norm(rng.random(50) * 7 + 3)
    assert v.min() == 0.0 and 0.99 < v.max() < 1.0


def check_sensitivity_branches():
    """Eq. (sensitivity): one branch is its own normalized score (not halved by the absent
    branch), two branches average, no branch gives no score."""
    rng = np.random.default_rng(5)
    cam = rng.standard_normal((6, 3, 4)) * np.arange(1, 7)[:, None, None]
    act = rng.standard_normal((6, 3, 4)) * np.arange(6, 0, -1)[:, None, None]
    n_cam = O.minmax_norm(O.control_rms(cam))
    n_act = O.minmax_norm(O.control_rms(act))
    assert np.allclose(O.sensitivity([cam]), n_cam)
    assert np.allclose(O.sensitivity([cam, act]), 0.5 * (n_cam + n_act))
    assert O.sensitivity([]) is None
    d = O.sensitivity([cam, act])
    assert d.min() >= 0.0 and d.max() <= 1.0


def check_frame_selection_worked_example():
    """Eqs. (debt), (score), TopK_f worked by hand for N_cur = 4, K_f = 2 (H_cov = 2):
    ages (0, 1, 2, 0) with anchors {0, 3} -> h = (0, 2, 3, 0), D = (0, 1, 1.5, 0);
    one branch with r = (1, 3, 2, 1) -> Norm = (0, 1, 0.5, 0) (eps = 0);
    S = d + 0.5 D = (0, 1.5, 1.25, 0) -> anchors {1, 2}."""
    delta = np.array([1.0, 3.0, 2.0, 1.0])[:, None] * np.ones((4, 6))
    anchors, h, S = O.select_frames([delta], [0, 1, 2, 0], [1, 0, 0, 1], 2, eps=0.0)
    assert list(h) == [0, 2, 3, 0]
    assert np.allclose(S, [0.0, 1.5, 1.25, 0.0])
    assert list(anchors) == [1, 2]
    # without a fresh response only the debt term: S = (0, 0.5, 0.75, 0) -> {1, 2} as well
    anchors, _, S = O.select_frames([], [0, 1, 2, 0], [1, 0, 0, 1], 2)
    assert np.allclose(S, [0.0, 0.5, 0.75, 0.0]) and list(anchors) == [1, 2]
    # ties go to the lower frame index: equal ages, no response -> the first K_f frames
    anchors, _, _ = O.select_frames([], [4, 4, 4, 4, 4], [0] * 5, 2)
    assert list(anchors) == [0, 1]
    # H_cov = ceil(5 / 2) = 3: ages (2, 0, 0, 0, 0), anchors {} -> D_0 = 3 / 3 = 1
    _, h, S = O.select_frames([], [2, 0, 0, 0, 0], [0] * 5, 2)
    assert np.allclose(S, 0.5 * h / 3.0) and S[0] == 0.5


def check_frame_selection_brute_force():
    """TopK_f against enumeration of every K_f-subset (largest score sum, ties to the
    lexicographically smallest index set), including all-frames and tied scores."""
    import itertools
    rng = np.random.default_rng(21)
    for trial in range(40):
        N = int(rng.integers(2, 8))
        K = int(rng.integers(1, N + 2))
        ages = rng.integers(0, 4, N)
        mask = rng.random(N) < 0.4
        deltas = [rng.standard_normal((N, 5)) * rng.integers(1, 3, N)[:, None]
                  for _ in range(int(rng.integers(0, 3)))]
        if trial % 5 == 0:
            deltas = []                                   # debt only: many ties
        anchors, h, S = O.select_frames(deltas, ages, mask, K)
        Ke = min(K, N)
        best = None
        for sub in itertools.combinations(range(N), Ke):
            key = (-round(sum(S[list(sub)]), 12), sub)
            if best is None or key < best:
                best = key
        assert tuple(anchors) == best[1], (anchors, best)
        assert len(anchors) == Ke and np.all(np.diff(anchors) > 0)




# ----------------------------------------------------------------------------------------------
# Output projection and anchor FFN
# ----------------------------------------------------------------------------------------------

def check_gelu_tanh_values():
    """The tanh form at printed values of 0.5 x (1 + tanh(sqrt(2/pi)(x + 0.044715 x^3))):
    gelu(1) = 0.8411919906, gelu(-1) = -0.1588080094, gelu(0) = 0, odd-part identity
    gelu(x) - gelu(-x) = x, and it lies within 1e-3 of the erf form on [-4, 4]."""
    assert abs(O.gelu_tanh(1.0) - 0.8411919906082768) < 1e-12
    assert abs(O.gelu_tanh(-1.0) + 0.15880800939172324) < 1e-12
    assert O.gelu_tanh(0.0) == 0.0
    x = np.linspace(-6, 6, 101)
    assert np.allclose(O.gelu_tanh(x) - O.gelu_tanh(-x), x, atol=1e-12)
    erf_form = 0.5 * x * (1.0 + scipy.special.erf(x / np.sqrt(2.0)))
    assert np.max(np.abs(O.gelu_tanh(x[np.abs(x) <= 4]) - erf_form[np.abs(x) <= 4])) < 1e-3


def check_linear_and_ffn_loops():
    """linear and anchor_ffn against explicit loops over every output (tiny sizes), reading
    only the anchor frames."""
    rng = np.random.default_rng(9)
    F, S, D, Dff = 4, 3, 5, 7
    x = rng.standard_normal((F, S, D))
    w1, b1 = rng.standard_normal((Dff, D)), rng.standard_normal(Dff)
    w2, b2 = rng.standard_normal((D, Dff)), rng.standard_normal(D)
    anchors = [0, 2]
    y = O.anchor_ffn(x, anchors, w1, b1, w2, b2)
    assert y.shape == (2, S, D)
    for ia, a in enumerate(anchors):
        for s in range(S):
            hid = []
            for j in range(Dff):
                acc = b1[j]
                for c in range(D):
                    acc += x[a, s, c] * w1[j, c]
                hid.append(0.5 * acc * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (acc + 0.044715 * acc ** 3))))
            for o in range(D):
                acc = b2[o]
                for j in range(Dff):
                    acc += hid[j] * w2[o, j]
                assert abs(y[ia, s, o] - acc) < 1e-10
    wsq = rng.standard_normal((D, D))            # a square weight (W_O): out = x W^T
    ysq = O.linear(x[0], wsq)
    for s_ in range(S):
        for o in range(D):
            assert abs(ysq[s_, o] - sum(x[0, s_, c] * wsq[o, c] for c in range(D))) < 1e-10
    x2 = x.copy()
    x2[1] += 100.0
    x2[3] -= 7.0                                   # skipped frames are not read
    assert np.array_equal(O.anchor_ffn(x2, anchors, w1, b1, w2, b2), y)


def check_projected_block_step_identity():
    """With W_O = I and no bias the projected block step equals the plain one (Eq. block)."""
    from synthetic import workloads as W
    wl = W.TINY
    inp = W.block_step_inputs(wl)
    D = wl.H * wl.d
    p = O.ParParams(band_radius=wl.band_radius)
    idx, Oa, r = O.block_step(inp, wl.K, wl.grid, p)
    _, _, r2 = O.block_step_projected(inp, wl.K, wl.grid, np.eye(D), None, p, idx=idx, O=Oa)
    assert np.allclose(r, r2, atol=1e-12)




# ----------------------------------------------------------------------------------------------
# Paper-granularity history blocks: (1, 8, 8) token blocks, partial blocks, K = ceil(0.2 M)
# ----------------------------------------------------------------------------------------------

def check_spatial_blocks_partition():
    """Blocks cover every token of every history frame exactly once; full blocks hold 64
    tokens, edge blocks h x w with h = Hg mod 8 or 8 and w = Wg mod 8 or 8; the count is
    F * ceil(Hg / 8) * ceil(Wg / 8)."""
    F, Hg, Wg = 2, 30, 52
    bl = O.spatial_blocks(F, Hg, Wg)
    assert len(bl) == F * 4 * 7
    for f in range(F):
        toks = np.concatenate([t for g, t in bl if g == f])
        assert np.array_equal(np.sort(toks), np.arange(Hg * Wg))
    sizes = sorted({len(t) for _, t in bl})
    assert sizes == sorted([6 * 4, 6 * 8, 8 * 4, 64])
    f, t = bl[7 * 3 + 6]                 # frame 0, last block row and column: 6 x 4 tokens
    assert f == 0 and list(t) == [y * Wg + x for y in range(24, 30) for x in range(48, 52)]


def check_spatial_blocks_reduce_to_token_ranges():
    """With an 8-token-wide history grid a (1, 8, 8) block is 64 consecutive tokens, so routing
    and attention over the spatial blocks equal the token-range forms with B_v = 64."""
    rng = np.random.default_rng(13)
    N, S, H, d = 2, 24, 2, 16
    Fh, Hg, Wg = 3, 24, 8                 # 3 frames x 3 blocks of 64 tokens
    q = rng.standard_normal((N, S, H, d))
    kc, vc = rng.standard_normal((N, S, H, d)), rng.standard_normal((N, S, H, d))
    kf = rng.standard_normal((Fh, Hg * Wg, H, d))
    vf = rng.standard_normal((Fh, Hg * Wg, H, d))
    bl = O.spatial_blocks(Fh, Hg, Wg)
    kb, vb = O.gather_blocks(kf, bl), O.gather_blocks(vf, bl)
    krange = kf.reshape(Fh * 3, 64, H, d)
    vrange = vf.reshape(Fh * 3, 64, H, d)
    a = O.pooled_routing(q, [0, 1], kb, vb)
    b = O.pooled_routing(q, [0, 1], krange, vrange)
    assert np.allclose(a.u, b.u, rtol=1e-12, atol=1e-14)
    idx = O.topk_blocks(a.u, 4)
    oa = O.routed_attention(q, kc, vc, kb, vb, [0, 1], idx)
    ob = O.routed_attention(q, kc, vc, krange, vrange, [0, 1], idx)
    assert np.allclose(oa, ob, rtol=1e-12, atol=1e-14)


def check_partial_block_statistics():
    """A truncated block pools over its own tokens only (no padding): brute-force means of an
    edge block; attention over it equals attention over exactly its tokens."""
    rng = np.random.default_rng(17)
    Hg, Wg, H, d = 10, 11, 1, 4
    kf = rng.standard_normal((1, Hg * Wg, H, d))
    bl = O.spatial_blocks(1, Hg, Wg)
    f, tok = bl[-1]                      # rows 8..9, columns 8..10: 6 tokens
    assert len(tok) == 6
    blk = O.gather_blocks(kf, bl)[-1]
    ref = np.zeros((H, d))
    for y in (8, 9):
        for x in (8, 9, 10):
            ref += kf[0, y * Wg + x]
    ref /= 6.0
    q = rng.standard_normal((1, 3, H, d))
    r = O.pooled_routing(q, [0], O.gather_blocks(kf, bl), O.gather_blocks(kf, bl))
    assert np.allclose(r.kbar[-1], ref, atol=1e-14)
    assert blk.shape[0] == 6
    assert O.paper_budget(448) == 90 and O.paper_budget(10) == 2 and O.paper_budget(1) == 1


ALL_CHECKS = [v for k, v in sorted(globals().items()) if k.startswith("check_")]

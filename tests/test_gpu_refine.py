"""Reconstruction-coupled routing refinement (Alg. routing, App. B.3) on the GPU against the
oracle.  The oracle is fed the GPU's own omission scores u, so the comparison isolates the
best-response passes: block sets must match exactly for every head whose decisions the oracle
does not flag as ambiguous (a gain within 1e-4 of the acceptance threshold, or a near tie at
the TopK boundary of a gain vector); for the rest the result must be a valid fixed-budget mask
set whose objective does not exceed the TopK initialisation's."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import workloads as W
from tests.gpu_util import to_dev, to_host
from tests.test_gpu_route import _inputs

pytestmark = pytest.mark.gpu

PAPER = dict(passes=2, lambda_anc=1.0, lambda_rec=1.0, tol=1e-6)


def _mask(idx, M):
    x = np.zeros((idx.shape[0], M))
    for i in range(idx.shape[0]):
        x[i, idx[i]] = 1.0
    return x


def check_refined(idx_gpu, u, anchors, n_frames, K, refine, candidates=None):
    """Compare [K_f, H, K_eff] refined indices with the oracle per head (candidates: optional
    [K_f, H, M_c] fixed sets); returns (#heads the refinement changed, #ambiguous heads)."""
    Kf, H, M = u.shape
    keff = min(K, M)
    changed = amb = 0
    for h in range(H):
        uh = u[:, h, :].astype(np.float64)
        ch = None if candidates is None else candidates[:, h, :]
        ref, info = O.coupled_routing(uh, anchors, n_frames, K, passes=refine["passes"],
                                      lam_anc=refine["lambda_anc"], lam_rec=refine["lambda_rec"],
                                      tol=refine["tol"], with_info=True, candidates=ch)
        g = idx_gpu[:, h, :]
        assert g.shape == (Kf, keff)
        for i in range(Kf):
            assert np.all(np.diff(g[i]) > 0) and g[i].min() >= 0 and g[i].max() < M
            if ch is not None:
                assert set(g[i].tolist()) <= set(ch[i].tolist())
        changed += int(not np.array_equal(ref, O.topk_blocks(uh, K, candidates=ch)))
        if not info["ambiguous"]:
            assert np.array_equal(g, ref), (h, g, ref)
        else:
            amb += 1
            co = info["coefficients"]
            j_init = info["trace"][0]
            j_gpu = O.routing_objective(uh, _mask(g, M), co, refine["lambda_anc"],
                                        refine["lambda_rec"])
            assert j_gpu <= j_init * (1 + 1e-5) + 1e-12
    return changed, amb


@pytest.mark.parametrize("dtype,d", [("bf16", 128), ("f32", 64)])
def test_refine_small(lib, dtype, d):
    N, S, H, M, Bv, K = 16, 40, 6, 40, 24, 8
    anchors = [0, 3, 7, 12, 15]
    q, k, v = _inputs(70 + d, N, S, H, d, M, Bv, dtype)
    idx, u = lib.cast_route_topk(to_dev(q, dtype), anchors, to_dev(k, dtype), to_dev(v, dtype),
                                 K, want_u=True, refine=PAPER)
    torch.cuda.synchronize()
    changed, amb = check_refined(idx.cpu().numpy(), to_host(u), anchors, N, K, PAPER)
    assert amb < H


@pytest.mark.parametrize("M,anchors", [(32, [0, 2, 4, 6, 8, 10, 12, 15]),
                                       (20, [0, 1, 3, 5, 6, 8, 10, 11, 13, 15]),
                                       (7, [2, 9])])
def test_refine_small_histories(lib, M, anchors):
    """Short histories (one warp's width of blocks and fewer) with many anchors (8 and 10:
    every interior interval and both boundary sets) and with two anchors (both boundary sets
    on the one pair)."""
    N, S, H, d, Bv, K = 16, 24, 4, 64, 16, 3
    q, k, v = _inputs(110 + M, N, S, H, d, M, Bv, "f32")
    idx, u = lib.cast_route_topk(to_dev(q, "f32"), anchors, to_dev(k, "f32"), to_dev(v, "f32"),
                                 K, want_u=True, refine=PAPER)
    torch.cuda.synchronize()
    changed, amb = check_refined(idx.cpu().numpy(), to_host(u), anchors, N, K, PAPER)
    assert amb < H


@pytest.mark.parametrize("passes", [1, 2, 5])
def test_refine_passes_and_weights(lib, passes):
    N, S, H, d, M, Bv, K = 12, 30, 4, 128, 24, 16, 5
    anchors = [1, 4, 6, 10]
    q, k, v = _inputs(90 + passes, N, S, H, d, M, Bv, "bf16")
    dq, dk, dv = (to_dev(x, "bf16") for x in (q, k, v))
    for lam_anc, lam_rec in ((1.0, 1.0), (0.5, 2.0), (1.0, 0.0)):
        ref = dict(passes=passes, lambda_anc=lam_anc, lambda_rec=lam_rec, tol=1e-6)
        idx, u = lib.cast_route_topk(dq, anchors, dk, dv, K, want_u=True, refine=ref)
        torch.cuda.synchronize()
        check_refined(idx.cpu().numpy(), to_host(u), anchors, N, K, ref)
        if lam_rec == 0.0:
            # no coupling: the best response is TopK(u), the initialisation
            assert np.array_equal(idx.cpu().numpy(), lib.cast_route_topk(dq, anchors, dk, dv, K)
                                  .cpu().numpy())


def test_refine_budget_edge_cases(lib):
    N, S, H, d, M, Bv = 6, 20, 2, 64, 9, 16
    anchors = [0, 2, 5]
    q, k, v = _inputs(5, N, S, H, d, M, Bv, "f32")
    dq, dk, dv = (to_dev(x, "f32") for x in (q, k, v))
    for K in (1, M - 1, M, M + 3):
        idx = lib.cast_route_topk(dq, anchors, dk, dv, K, refine=PAPER)
        plain = lib.cast_route_topk(dq, anchors, dk, dv, K)
        torch.cuda.synchronize()
        assert idx.shape == (3, H, min(K, M))
        if K >= M:   # nothing to choose: every block routed, refinement skipped
            assert np.array_equal(idx.cpu().numpy(), plain.cpu().numpy())


@pytest.mark.parametrize("wl", [W.MG, W.HY], ids=lambda w: w.name)
def test_refine_full_size(lib, wl):
    inp = W.block_step_inputs(wl)
    dk = (lambda x: to_dev(x, "bf16"))
    idx, u = lib.cast_route_topk(dk(inp["q"]), list(wl.anchors), dk(inp["k_hist"]),
                                 dk(inp["v_hist"]), wl.K, want_u=True, refine=PAPER)
    torch.cuda.synchronize()
    changed, amb = check_refined(idx.cpu().numpy(), to_host(u), list(wl.anchors), wl.n_cur,
                                 wl.K, PAPER)
    assert changed > 0          # the workload exercises the coupling
    assert amb <= wl.H // 4


def test_refine_stress_long_history(lib):
    w = W.STRESS
    inp = W.stress_inputs(w)
    dk = (lambda x: to_dev(x, "bf16"))
    q, kh, vh = dk(inp["q"]), dk(inp["k_hist"]), dk(inp["v_hist"])
    anchors = list(range(w.n_cur))
    for K in w.Ks:
        idx, u = lib.cast_route_topk(q, anchors, kh, vh, K, want_u=True, refine=PAPER)
        torch.cuda.synchronize()
        check_refined(idx.cpu().numpy(), to_host(u), anchors, w.n_cur, K, PAPER)


def test_block_step_routes_with_refinement(lib):
    wl = W.MG
    inp = W.block_step_inputs(wl)
    dk = (lambda x: to_dev(x, "bf16"))
    N, S, H, d = inp["q"].shape
    q, kc, vc, kh, vh = (dk(inp[k]) for k in ("q", "k_cur", "v_cur", "k_hist", "v_hist"))
    r_out = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device="cuda")
    idx = torch.empty((len(wl.anchors), H, wl.K), dtype=torch.int32, device="cuda")
    lib.cast_block_step(q, kc, vc, list(wl.anchors), kh, vh, wl.K, wl.grid, r_out, idx_out=idx,
                        refine=PAPER)
    ref = lib.cast_route_topk(q, list(wl.anchors), kh, vh, wl.K, refine=PAPER)
    torch.cuda.synchronize()
    lib.cast_check_device()
    assert np.array_equal(idx.cpu().numpy(), ref.cpu().numpy())

"""Routing kernels (cast_route_topk) against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import TOPK_GAP, to_dev, to_host

pytestmark = pytest.mark.gpu


def _inputs(seed, N, S, H, d, M, Bv, dtype):
    ss = np.random.SeedSequence(seed)
    a, b, c = ss.spawn(3)
    q = G.tokens_with_offsets(a, N, S, H, d, 1.0)
    k = G.tokens_with_offsets(b, M, Bv, H, d, 1.0)
    v = G.tokens_with_offsets(c, M, Bv, H, d, 1.0)
    if dtype == "bf16":
        q, k, v = G.round_bf16(q), G.round_bf16(k), G.round_bf16(v)
    return q, k, v


def check_idx(idx_gpu, score_ref, K):
    """Sets match wherever the oracle's relative gap at the K boundary exceeds TOPK_GAP;
    elsewhere only blocks outside the ambiguous band must agree.  Returns #ambiguous."""
    ref = O.topk_blocks(score_ref, K)
    gap = O.topk_margin(score_ref, K)
    amb = 0
    for r in np.ndindex(ref.shape[:-1]):
        g = idx_gpu[r]
        assert np.all(np.diff(g) > 0), "indices not strictly ascending"
        if gap[r] > TOPK_GAP:
            assert np.array_equal(g, ref[r]), (r, g, ref[r])
        else:
            amb += 1
            s = score_ref[r]
            kth = np.sort(s)[::-1][K - 1]
            lo, hi = kth - TOPK_GAP * abs(kth), kth + TOPK_GAP * abs(kth)
            assert set(np.flatnonzero(s > hi)) <= set(g.tolist())
            assert not (set(np.flatnonzero(s < lo)) & set(g.tolist()))
    return amb


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("d", [64, 128])
def test_route_small(lib, dtype, d):
    N, S, H, M, Bv, K = 3, 50, 3, 7, 37, 3
    q, k, v = _inputs(10 + d, N, S, H, d, M, Bv, dtype)
    anchors = [0, 2]
    idx, u, (qb, kb, vb) = lib.cast_route_topk(to_dev(q, dtype), anchors, to_dev(k, dtype),
                                                to_dev(v, dtype), K, want_u=True, want_pooled=True)
    torch.cuda.synchronize()
    rt = O.pooled_routing(q, anchors, k, v)
    np.testing.assert_allclose(to_host(qb), rt.qbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(kb), rt.kbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(vb), rt.vbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(u), rt.u, rtol=2e-4, atol=1e-7 * rt.u.max())
    amb = check_idx(idx.cpu().numpy(), rt.u, K)
    assert amb == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_route_bulk_pooling(lib, dtype):
    """Long contiguous segments (at least 1 MB per pooling CTA in both launches), which the
    pooling streams through its bulk-copy ring: pooled means, u and TopK against the oracle."""
    N, S, H, d, M, Bv, K = 3, 2048, 12, 128, 4, 4096, 2
    q, k, v = _inputs(31, N, S, H, d, M, Bv, dtype)
    anchors = [0, 2]
    idx, u, (qb, kb, vb) = lib.cast_route_topk(to_dev(q, dtype), anchors, to_dev(k, dtype),
                                                to_dev(v, dtype), K, want_u=True, want_pooled=True)
    torch.cuda.synchronize()
    lib.cast_check_device()
    rt = O.pooled_routing(q, anchors, k, v)
    np.testing.assert_allclose(to_host(qb), rt.qbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(kb), rt.kbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(vb), rt.vbar, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(to_host(u), rt.u, rtol=2e-4, atol=1e-7 * rt.u.max())
    check_idx(idx.cpu().numpy(), rt.u, K)


def test_route_gram_projection(lib):
    """GPU with G = P^T P equals the oracle's literal ||P delta||^2 (Eq. omission)."""
    N, S, H, d, M, Bv, K = 2, 64, 2, 64, 9, 40, 4
    q, k, v = _inputs(21, N, S, H, d, M, Bv, "bf16")
    P = np.random.default_rng(5).standard_normal((H, d, d)) / np.sqrt(d)
    gram = np.einsum("hod,hoe->hde", P, P).astype(np.float32)
    idx, u = lib.cast_route_topk(to_dev(q, "bf16"), [1], to_dev(k, "bf16"), to_dev(v, "bf16"), K,
                                 gram=torch.from_numpy(gram).cuda(), want_u=True)
    torch.cuda.synchronize()
    rt = O.pooled_routing(q, [1], k, v, proj=P)
    np.testing.assert_allclose(to_host(u), rt.u, rtol=5e-4, atol=1e-7 * rt.u.max())
    check_idx(idx.cpu().numpy(), rt.u, K)


def test_route_similarity_mode(lib):
    N, S, H, d, M, Bv, K = 2, 33, 2, 128, 11, 20, 5
    q, k, v = _inputs(22, N, S, H, d, M, Bv, "bf16")
    idx, s = lib.cast_route_topk(to_dev(q, "bf16"), [0, 1], to_dev(k, "bf16"), to_dev(v, "bf16"), K,
                                 mode=lib.ROUTE_SIMILARITY, want_u=True)
    torch.cuda.synchronize()
    rt = O.pooled_routing(q, [0, 1], k, v)
    np.testing.assert_allclose(to_host(s), rt.s, rtol=1e-4, atol=1e-5)
    check_idx(idx.cpu().numpy(), rt.s, K)


def test_route_bypass_keeps_all_blocks(lib):
    q, k, v = _inputs(23, 2, 16, 2, 64, 5, 8, "bf16")
    idx = lib.cast_route_topk(to_dev(q, "bf16"), [0, 1], to_dev(k, "bf16"), to_dev(v, "bf16"), 9)
    torch.cuda.synchronize()
    assert idx.shape == (2, 2, 5)
    assert np.array_equal(idx.cpu().numpy(), np.broadcast_to(np.arange(5), (2, 2, 5)))


@pytest.mark.parametrize("K", [4, 8, 16, 32])
def test_route_stress_full_size(lib, K, stress_inputs):
    """Long-history stress workload at full size (128 blocks of 3520 tokens, 24 heads)."""
    inp = stress_inputs
    idx, u = lib.cast_route_topk(inp["dev"]["q"], list(inp["anchors"]), inp["dev"]["k_hist"],
                                 inp["dev"]["v_hist"], K, want_u=True)
    torch.cuda.synchronize()
    u_ref = inp["routing"].u
    np.testing.assert_allclose(to_host(u), u_ref, rtol=1e-3, atol=1e-6 * u_ref.max())
    amb = check_idx(idx.cpu().numpy(), u_ref, K)
    if K <= 8:
        assert amb == 0


@pytest.fixture(scope="module")
def stress_inputs():
    import oracle.cast_oracle as O  # noqa: F811
    w = W.STRESS
    inp = W.stress_inputs(w)
    dev = {k: to_dev(inp[k], "bf16") for k in ("q", "k_hist", "v_hist")}
    anchors = [int(a) for a in inp["anchors"]]
    # oracle pooled statistics block by block (float64), then Eqs. pooled / omission
    q = inp["q"]
    qbar = np.stack([q[a].astype(np.float64).mean(axis=0) for a in anchors])
    kbar = np.stack([inp["k_hist"][m].astype(np.float64).mean(axis=0) for m in range(w.M)])
    vbar = np.stack([inp["v_hist"][m].astype(np.float64).mean(axis=0) for m in range(w.M)])
    rt = O.pooled_routing(qbar[:, None], list(range(len(anchors))), kbar[:, None], vbar[:, None])
    return {"dev": dev, "anchors": anchors, "routing": rt}


WIDE_CASES = [
    # name, d, dtype, M, B_v, K, anchors, N, extra
    ("refine_d128", 128, "bf16", 448, 16, 90, [0, 2, 4, 6], 8, {"refine": True}),
    ("refine_d64_f32", 64, "f32", 1000, 6, 200, [0, 3, 7, 12, 15], 16, {"refine": True}),
    ("topk_k1", 128, "bf16", 300, 8, 1, [1, 2], 3, {}),
    ("keep_all", 64, "bf16", 300, 8, 300, [0, 2], 3, {}),
    ("similarity", 128, "bf16", 300, 8, 7, [0, 1], 2, {"mode": 1}),
    ("gram", 128, "bf16", 260, 8, 50, [0, 2], 3, {"gram": True}),
    ("candidates", 128, "bf16", 500, 8, 100, [0, 3, 5], 6, {"refine": True, "Mc": 150}),
]


@pytest.mark.parametrize("case", WIDE_CASES, ids=lambda c: c[0])
def test_route_wide(lib, case):
    """Many history blocks: the per-head statistics spread over a cluster of CTAs and the
    radix-select TopK / refinement (block means too large for one CTA's shared memory)."""
    from tests.test_gpu_refine import PAPER, check_refined
    name, d, dtype, M, Bv, K, anchors, N, extra = case
    H, S = 2, 40
    q, k, v = _inputs(500 + M + d, N, S, H, d, M, Bv, dtype)
    kw = {}
    P = None
    if extra.get("gram"):
        P = np.random.default_rng(6).standard_normal((H, d, d)) / np.sqrt(d)
        kw["gram"] = torch.from_numpy(np.einsum("hod,hoe->hde", P, P).astype(np.float32)).cuda()
    if "mode" in extra:
        kw["mode"] = extra["mode"]
    if extra.get("refine"):
        kw["refine"] = PAPER
    cand = None
    if "Mc" in extra:
        rng = np.random.default_rng(M)
        cand = np.stack([[rng.permutation(M)[:extra["Mc"]] for _ in range(H)]
                         for _ in anchors]).astype(np.int32)
        kw["candidates"] = torch.from_numpy(cand).cuda()
    idx, u = lib.cast_route_topk(to_dev(q, dtype), anchors, to_dev(k, dtype), to_dev(v, dtype), K,
                                 want_u=True, **kw)
    torch.cuda.synchronize()
    lib.cast_check_device()
    rt = O.pooled_routing(q, anchors, k, v, proj=P)
    ug = to_host(u)
    score = rt.u if extra.get("mode") != 1 else rt.s
    np.testing.assert_allclose(ug, score, rtol=5e-4, atol=1e-6 * np.abs(score).max())
    g = idx.cpu().numpy()
    assert g.shape == (len(anchors), H, min(K, M))
    if extra.get("refine"):
        changed, amb = check_refined(g, ug, anchors, N, K, PAPER, candidates=cand)
        assert amb < H
    else:
        check_idx(g, score, min(K, M))

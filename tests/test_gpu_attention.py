"""Routed anchor attention (cast_anchor_attention, tcgen05 kernel) against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import ATTN_REL_MAX, to_dev, to_host

pytestmark = pytest.mark.gpu


def _inputs(seed, N, S, H, d, M, Bv):
    ss = np.random.SeedSequence(seed)
    parts = ss.spawn(5)
    q = G.round_bf16(G.tokens_with_offsets(parts[0], N, S, H, d, 0.5))
    kc = G.round_bf16(G.tokens_with_offsets(parts[1], N, S, H, d, 0.5))
    vc = G.round_bf16(G.tokens_with_offsets(parts[2], N, S, H, d, 0.5))
    kh = G.round_bf16(G.tokens_with_offsets(parts[3], M, Bv, H, d, 0.5))
    vh = G.round_bf16(G.tokens_with_offsets(parts[4], M, Bv, H, d, 0.5))
    return q, kc, vc, kh, vh


def _rel_err(gpu, ref):
    return float(np.max(np.abs(gpu - ref)) / np.max(np.abs(ref)))


CASES = [
    # N, S, H, d, M, Bv, K, anchors, out dtype
    (3, 200, 2, 64, 4, 150, 2, (0, 2), torch.float32),
    (3, 200, 2, 128, 4, 150, 2, (0, 2), torch.float32),
    (2, 128, 1, 128, 3, 128, 3, (1,), torch.bfloat16),
    (4, 64, 2, 64, 4, 64, 2, (0, 3), torch.float32),        # the tiny block-step shape
    (2, 300, 3, 128, 5, 1000, 3, (0, 1), torch.bfloat16),
    (3, 77, 2, 128, 0, 1, 0, (0, 2), torch.float32),        # no history
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"N{c[0]}S{c[1]}H{c[2]}d{c[3]}M{c[4]}Bv{c[5]}K{c[6]}")
def test_attention_small(lib, case):
    N, S, H, d, M, Bv, K, anchors, odt = case
    q, kc, vc, kh, vh = _inputs(100 + S + d, N, S, H, d, max(M, 1), Bv)
    rng = np.random.default_rng(S)
    idx = np.stack([[rng.permutation(M)[:K] for _ in range(H)] for _ in anchors]).astype(np.int32) \
        if M else np.zeros((len(anchors), H, 0), np.int32)
    dk = (lambda x: to_dev(x, "bf16"))
    o, lse = lib.cast_anchor_attention(dk(q), dk(kc), dk(vc), list(anchors),
                                       dk(kh) if M else None, dk(vh) if M else None,
                                       torch.from_numpy(idx).cuda() if M else None,
                                       out_dtype=odt, want_lse=True)
    torch.cuda.synchronize()
    ref, lse_ref = O.routed_attention(q, kc, vc, kh, vh, list(anchors), idx if M else None,
                                      with_lse=True)
    ref = ref.reshape(len(anchors), S, H * d)
    err = _rel_err(to_host(o), ref)
    assert err <= ATTN_REL_MAX, err
    np.testing.assert_allclose(to_host(lse), lse_ref, atol=2e-2)


def test_attention_all_history_equals_dense(lib):
    """Routing every block equals dense attention over current + all history (oracle)."""
    N, S, H, d, M, Bv = 2, 130, 2, 128, 3, 129
    q, kc, vc, kh, vh = _inputs(7, N, S, H, d, M, Bv)
    idx = np.tile(np.arange(M, dtype=np.int32)[::-1], (1, H, 1))
    dk = (lambda x: to_dev(x, "bf16"))
    o = lib.cast_anchor_attention(dk(q), dk(kc), dk(vc), [1], dk(kh), dk(vh),
                                  torch.from_numpy(np.ascontiguousarray(idx)).cuda(),
                                  out_dtype=torch.float32)
    torch.cuda.synchronize()
    ref = O.routed_attention(q, kc, vc, kh, vh, [1], np.tile(np.arange(M), (1, H, 1)))
    assert _rel_err(to_host(o), ref.reshape(1, S, H * d)) <= ATTN_REL_MAX


@pytest.mark.parametrize("wl", [W.MG, W.HY], ids=lambda w: w.name)
def test_attention_full_size_sampled_rows(lib, wl):
    """Full-size block-step attention shapes; every head of every anchor, a sample of query
    rows (first, ragged last tile, random) checked against the oracle."""
    inp = W.block_step_inputs(wl)
    dk = (lambda x: to_dev(x, "bf16"))
    rng = np.random.default_rng(wl.seed)
    Kf = len(wl.anchors)
    idx = np.stack([[np.sort(rng.permutation(wl.M)[:wl.K]) for _ in range(wl.H)]
                    for _ in range(Kf)]).astype(np.int32)
    o = lib.cast_anchor_attention(dk(inp["q"]), dk(inp["k_cur"]), dk(inp["v_cur"]),
                                  list(wl.anchors), dk(inp["k_hist"]), dk(inp["v_hist"]),
                                  torch.from_numpy(idx).cuda(), out_dtype=torch.float32)
    torch.cuda.synchronize()
    S = wl.S
    rows = np.unique(np.concatenate([[0, 1, 127, 128, S - 1], rng.integers(0, S, 11)]))
    ref = O.routed_attention(inp["q"], inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                             list(wl.anchors), idx, rows=rows)
    g = to_host(o).reshape(Kf, S, wl.H, wl.d)[:, rows]
    r = ref[:, rows]
    assert _rel_err(g, r) <= ATTN_REL_MAX

"""Fixed candidate sets C_i (App. B.3) in cast_route_topk and cast_block_step against the
oracle: TopK and the coupled refinement choose within C_i, blocks outside stay omitted, and
bad candidate indices are reported by cast_check_device without a fault."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import workloads as W
from tests.gpu_util import to_dev, to_host
from tests.test_gpu_refine import PAPER, check_refined
from tests.test_gpu_route import _inputs, check_idx

pytestmark = pytest.mark.gpu


def _sets(seed, Kf, H, M, Mc):
    rng = np.random.default_rng(seed)
    c = np.stack([[rng.permutation(M)[:Mc] for _ in range(H)] for _ in range(Kf)])
    return c.astype(np.int32)


@pytest.mark.parametrize("Mc_extra", [0, 3, None])
def test_candidate_topk(lib, Mc_extra):
    N, S, H, d, M, Bv, K = 4, 40, 3, 128, 20, 16, 5
    anchors = [0, 2, 3]
    q, k, v = _inputs(31, N, S, H, d, M, Bv, "bf16")
    Mc = M if Mc_extra is None else K + Mc_extra
    c = _sets(7 + Mc, len(anchors), H, M, Mc)
    idx, u = lib.cast_route_topk(to_dev(q, "bf16"), anchors, to_dev(k, "bf16"), to_dev(v, "bf16"),
                                 K, want_u=True, candidates=torch.from_numpy(c).cuda())
    torch.cuda.synchronize()
    lib.cast_check_device()
    ug = to_host(u)
    rt = O.pooled_routing(q, anchors, k, v)
    np.testing.assert_allclose(ug, rt.u, rtol=2e-4, atol=1e-7 * rt.u.max())
    g = idx.cpu().numpy()
    restricted = np.where(O.candidate_mask(c, M, K), rt.u, -np.inf)
    check_idx(g, restricted, K)
    for r in np.ndindex(g.shape[:-1]):
        assert set(g[r].tolist()) <= set(c[r].tolist())


@pytest.mark.parametrize("Mc", [8, 13])
@pytest.mark.parametrize("M", [40, 24])
def test_candidate_refinement(lib, Mc, M):
    N, S, H, d, Bv, K = 16, 40, 6, 128, 24, 8
    anchors = [0, 3, 7, 12, 15]
    q, k, v = _inputs(72, N, S, H, d, M, Bv, "bf16")
    c = _sets(Mc, len(anchors), H, M, Mc)
    idx, u = lib.cast_route_topk(to_dev(q, "bf16"), anchors, to_dev(k, "bf16"), to_dev(v, "bf16"),
                                 K, want_u=True, refine=PAPER, candidates=torch.from_numpy(c).cuda())
    torch.cuda.synchronize()
    lib.cast_check_device()
    changed, amb = check_refined(idx.cpu().numpy(), to_host(u), anchors, N, K, PAPER, candidates=c)
    assert amb < H


def test_candidate_full_sets_equal_unrestricted(lib):
    """C_i = every block recovers the unrestricted routing (Alg. routing with M_c = M)."""
    wl = W.MG
    inp = W.block_step_inputs(wl)
    dk = (lambda x: to_dev(x, "bf16"))
    q, kh, vh = dk(inp["q"]), dk(inp["k_hist"]), dk(inp["v_hist"])
    an = list(wl.anchors)
    full = torch.from_numpy(_sets(1, len(an), wl.H, wl.M, wl.M)).cuda()
    a = lib.cast_route_topk(q, an, kh, vh, wl.K, refine=PAPER, candidates=full)
    b = lib.cast_route_topk(q, an, kh, vh, wl.K, refine=PAPER)
    torch.cuda.synchronize()
    assert np.array_equal(a.cpu().numpy(), b.cpu().numpy())


def test_candidate_block_step(lib):
    wl = W.MG
    inp = W.block_step_inputs(wl)
    dk = (lambda x: to_dev(x, "bf16"))
    N, S, H, d = inp["q"].shape
    q, kc, vc, kh, vh = (dk(inp[k]) for k in ("q", "k_cur", "v_cur", "k_hist", "v_hist"))
    an = list(wl.anchors)
    c = torch.from_numpy(_sets(2, len(an), H, wl.M, 9)).cuda()
    r_out = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device="cuda")
    idx = torch.empty((len(an), H, wl.K), dtype=torch.int32, device="cuda")
    lib.cast_block_step(q, kc, vc, an, kh, vh, wl.K, wl.grid, r_out, idx_out=idx, refine=PAPER,
                        candidates=c)
    ref = lib.cast_route_topk(q, an, kh, vh, wl.K, refine=PAPER, candidates=c)
    torch.cuda.synchronize()
    lib.cast_check_device()
    assert np.array_equal(idx.cpu().numpy(), ref.cpu().numpy())


@pytest.mark.parametrize("bad", ["repeated", "outside"])
def test_candidate_bad_index_is_reported(lib, bad):
    N, S, H, d, M, Bv, K = 3, 20, 2, 64, 10, 8, 3
    q, k, v = _inputs(3, N, S, H, d, M, Bv, "f32")
    c = _sets(4, 2, H, M, 5)
    c[1, 0, 2] = c[1, 0, 0] if bad == "repeated" else M + 3
    lib.cast_route_topk(to_dev(q, "f32"), [0, 2], to_dev(k, "f32"), to_dev(v, "f32"), K,
                        candidates=torch.from_numpy(c).cuda())
    with pytest.raises(lib.CastError) as e:
        lib.cast_check_device()
    assert e.value.status == lib.ERR_INVALID_ARG
    lib.cast_check_device()    # the record is cleared

"""Control-aware frame selection (cast_select_frames) against the CPU oracle: per-frame RMS of
the control updates, scores, refresh ages and the selected anchors (exact wherever the
oracle's gap at the K_f boundary exceeds the TopK tolerance), over single calls and a chain of
blocks that feeds each call's ages and mask into the next."""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W
from tests.gpu_util import TOPK_GAP, to_dev, to_host

pytestmark = pytest.mark.gpu


def _check(gpu, deltas, ages, mask, K_f, lam=0.5, eps=1e-8):
    anchors, ages_out, mask_out, rms, score = gpu
    ref_anchors, ref_h, ref_S = O.select_frames(deltas, ages, mask, K_f, lam, eps)
    assert np.array_equal(ages_out.cpu().numpy(), ref_h)
    if deltas:
        ref_r = np.stack([O.control_rms(dk) for dk in deltas])
        np.testing.assert_allclose(to_host(rms), ref_r, rtol=2e-5)
    np.testing.assert_allclose(to_host(score), ref_S, rtol=2e-5, atol=2e-6)
    got = anchors.cpu().numpy()
    assert len(got) == min(K_f, len(ages)) and np.all(np.diff(got) > 0)
    assert np.array_equal(np.flatnonzero(mask_out.cpu().numpy()), got)
    if O.selection_margin(ref_S, K_f) > TOPK_GAP:
        assert np.array_equal(got, ref_anchors), (got, ref_anchors)
    else:   # a near tie at the boundary: only clearly ranked frames must agree
        s = np.sort(ref_S)[::-1]
        kth = s[min(K_f, len(s)) - 1]
        band = TOPK_GAP * max(abs(kth), 1e-30)
        assert set(np.flatnonzero(ref_S > kth + band)) <= set(got.tolist())
        assert not (set(np.flatnonzero(ref_S < kth - band)) & set(got.tolist()))
    return got, ref_h


def _run(lib, deltas, ages, mask, K_f, dtype):
    dd = [to_dev(x, dtype) for x in deltas]
    a = torch.from_numpy(np.asarray(ages, np.int32)).cuda()
    m = torch.from_numpy(np.asarray(mask, np.uint8)).cuda()
    out = lib.cast_select_frames(dd, a, m, K_f, want_rms=True, want_score=True)
    torch.cuda.synchronize()
    return out


CASES = [
    # N_cur, S, D, branches, dtype, K_f
    (10, 64, 256, 2, "f32", 5),      # Matrix-Game: five of ten current frames
    (4, 64, 128, 2, "bf16", 2),      # HY-World: two of four
    (8, 40, 64, 1, "bf16", 3),       # one branch
    (6, 40, 64, 0, "f32", 3),        # no fresh response: debt only
    (5, 16, 64, 2, "f32", 7),        # K_f > N_cur: every frame
    (256, 8, 64, 2, "f32", 100),     # the frame maximum
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"N{c[0]}_S{c[1]}_D{c[2]}_b{c[3]}_{c[4]}_K{c[5]}")
def test_select_small(lib, case):
    N, S, D, nb, dt, K_f = case
    ss = np.random.SeedSequence(N * 31 + nb)
    sd, sa = ss.spawn(2)
    deltas = G.control_updates(sd, nb, N, S, D)
    if dt == "bf16":
        deltas = [G.round_bf16(x) for x in deltas]
    rng = np.random.default_rng(N + D)
    ages = rng.integers(0, 5, N).astype(np.int32)
    mask = (rng.random(N) < 0.5).astype(np.uint8)
    _check(_run(lib, deltas, ages, mask, K_f, dt), deltas, ages, mask, K_f)


def test_select_ties_go_to_lower_frames(lib):
    # equal ages, no response: every score ties, the first K_f frames are chosen
    out = _run(lib, [], np.full(9, 3, np.int32), np.zeros(9, np.uint8), 4, "f32")
    assert out[0].cpu().numpy().tolist() == [0, 1, 2, 3]
    # a constant response contributes zero: scores are the debt alone
    flat = [np.ones((9, 8, 16), np.float32) * 0.7]
    out = _run(lib, flat, np.arange(9, dtype=np.int32), np.zeros(9, np.uint8), 3, "f32")
    _check(out, flat, np.arange(9, dtype=np.int32), np.zeros(9, np.uint8), 3)
    assert out[0].cpu().numpy().tolist() == [6, 7, 8]


def test_select_chain_of_blocks(lib):
    """Three blocks in a row on the device: each call's ages and mask feed the next."""
    N, S, D, K_f = 10, 32, 64, 5
    ss = np.random.SeedSequence(77)
    ages = np.zeros(N, np.int32)
    mask = np.ones(N, np.uint8)          # the dense first block of an evaluation
    a_dev = torch.from_numpy(ages).cuda()
    m_dev = torch.from_numpy(mask).cuda()
    for blk, child in enumerate(ss.spawn(3)):
        deltas = G.control_updates(child, 2, N, S, D)
        dd = [to_dev(x, "f32") for x in deltas]
        out = lib.cast_select_frames(dd, a_dev, m_dev, K_f, want_rms=True, want_score=True)
        torch.cuda.synchronize()
        got, ref_h = _check(out, deltas, ages, mask, K_f)
        ages = ref_h.astype(np.int32)
        mask = np.zeros(N, np.uint8)
        mask[got] = 1
        a_dev, m_dev = out[1], out[2]


def test_select_full_size(lib):
    w = W.SELECT_MG
    deltas, ages, mask = W.select_inputs(w)
    _check(_run(lib, deltas, ages, mask, w.K_f, "bf16"), deltas, ages, mask, w.K_f)

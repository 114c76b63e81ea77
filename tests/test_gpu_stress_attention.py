"""Routed anchor attention at the long-history stress configuration against the oracle.

Four anchor frames of 44x80 tokens, 24 heads x 128, 128 history blocks of 3520 tokens
(450,560 history tokens), K in {4, 8, 16, 32}: each (anchor, head) attends to the whole
current chunk plus its K routed blocks, up to 36 x 3520 = 126,720 keys (Eq. block,
App. B.4).  The attention is fed the GPU's own routed blocks (cast_route_topk on the same
inputs); sampled query rows (the first and last rows, both sides of 128-row query-tile
boundaries, and random rows) of sampled heads are compared with the float64 oracle at
max |err| / max |ref| <= 2e-2.
"""
import numpy as np
import pytest
import torch

import oracle.cast_oracle as O
from synthetic import workloads as W
from tests.gpu_util import ATTN_REL_MAX, to_dev, to_host

pytestmark = pytest.mark.gpu

HEADS = (0, 11, 23)


@pytest.fixture(scope="module")
def stress():
    w = W.STRESS
    inp = W.stress_inputs(w)
    dev = {k: to_dev(inp[k], "bf16") for k in ("q", "k_cur", "v_cur", "k_hist", "v_hist")}
    rng = np.random.default_rng(w.seed)
    rows = np.unique(np.concatenate([[0, 127, 128, 255, 256, 3455, w.S - 1],
                                     rng.integers(0, w.S, 3)]))
    return {"w": w, "inp": inp, "dev": dev, "rows": rows}


@pytest.mark.parametrize("K", [4, 8, 16, 32])
def test_attention_stress_full_size(lib, stress, K):
    w, inp, dv, rows = stress["w"], stress["inp"], stress["dev"], stress["rows"]
    anchors = [int(a) for a in inp["anchors"]]
    idx = lib.cast_route_topk(dv["q"], anchors, dv["k_hist"], dv["v_hist"], K)
    o = lib.cast_anchor_attention(dv["q"], dv["k_cur"], dv["v_cur"], anchors, dv["k_hist"],
                                  dv["v_hist"], idx)
    torch.cuda.synchronize()
    lib.cast_check_device()
    idx_h = idx.cpu().numpy()
    assert idx_h.shape == (len(anchors), w.H, K)
    g = to_host(o).reshape(len(anchors), w.S, w.H, w.d)
    ref = O.routed_attention(inp["q"], inp["k_cur"], inp["v_cur"], inp["k_hist"], inp["v_hist"],
                             anchors, idx_h, rows=rows, heads=HEADS)
    for h in HEADS:
        gr, rr = g[:, rows, h], ref[:, rows, h]
        err = np.max(np.abs(gr - rr)) / np.max(np.abs(rr))
        assert err <= ATTN_REL_MAX, (K, h, err)

"""Host-side checks of the synthetic workloads of the paper-granularity history blocks: their
sizes follow the oracle's block definition and budget (App. C Tab. config, Tab. config_cast),
and the history-frame generator is seeded and carries the per-patch structure it states."""
import numpy as np

import bench
import oracle.cast_oracle as O
from synthetic import generators as G
from synthetic import workloads as W


def test_paper_granularity_workload_sizes():
    for wl in (W.MG64, W.HY64):
        blocks = O.spatial_blocks(wl.hist_frames, *wl.grid)
        assert wl.M == len(blocks)
        assert wl.K == O.paper_budget(wl.M)
        assert wl.B_v == 64
        # the bench's per-block token counts (algorithmic FLOP of the attention scale point)
        assert bench._block_tokens(wl) == [len(t) for _, t in blocks]


def test_region_offsets_generator():
    ss = np.random.SeedSequence(3)
    a = G.frames_with_region_offsets(ss, 2, 11, 13, 2, 16, 2.0)
    b = G.frames_with_region_offsets(np.random.SeedSequence(3), 2, 11, 13, 2, 16, 2.0)
    assert a.shape == (2, 11, 13, 2, 16) and a.dtype == np.float32
    assert np.array_equal(a, b)
    # inside a patch the tokens share one offset: their spread is the N(0,1) noise alone,
    # while patch means spread with the offset scale
    patch = a[0, 0:8, 0:8, 0].reshape(64, 16)
    assert 0.8 < patch.std(axis=0).mean() < 1.2
    means = np.stack([a[f, y:y + 8, x:x + 8, 0].reshape(-1, 16).mean(axis=0)
                      for f in range(2) for y in (0, 8) for x in (0, 8)])
    assert means.std(axis=0).mean() > 1.2

"""Helpers for the GPU parity tests: move seeded numpy inputs to the device with the exact
bits the oracle sees, and the tolerances of the parity bar."""
from __future__ import annotations

import numpy as np
import torch

from synthetic import generators as G


def to_dev(x: np.ndarray, dtype: str, device="cuda"):
    """float32 numpy -> device tensor; bf16 uses the RN-even bits the oracle also sees."""
    if dtype == "bf16":
        bits = G.bf16_bits(x)
        return torch.from_numpy(bits.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(device)


def to_host(t: torch.Tensor) -> np.ndarray:
    return t.float().cpu().numpy().astype(np.float64)


# fp32 PAR: within 1e-4 of the frame residual's RMS (per target frame)
PAR_F32_REL_RMS = 1e-4
# bf16 attention: max |err| / max |ref| below 2e-2
ATTN_REL_MAX = 2e-2
# routing: blocks must match wherever the oracle's relative gap at the K boundary exceeds 1e-3
TOPK_GAP = 1e-3


def par_check(gpu, ref, targets, dtype, info=None, tiles=None, Hg=None, Wg=None, th=8, tw=8,
              excluded_tiles=()):
    """Asserts the PAR parity bar on every target frame; returns the worst ratio err / tol."""
    worst = 0.0
    for t in targets:
        g = gpu[t]
        r = ref[t]
        rms = float(np.sqrt(np.mean(r ** 2)))
        delta = PAR_F32_REL_RMS * rms
        if dtype == "bf16":
            tol = 2.0 ** -8 * (np.abs(r) + delta) + delta
        else:
            tol = np.full_like(r, delta)
        err = np.abs(g - r)
        mask = np.ones(r.shape[:2], dtype=bool)
        for (y0, x0) in excluded_tiles:
            mask[y0:y0 + th, x0:x0 + tw] = False
        ratio = (err / tol)[mask]
        if ratio.size:
            worst = max(worst, float(ratio.max()))
        assert ratio.size == 0 or ratio.max() <= 1.0, (
            f"frame {t}: max err {float(err[mask].max()):.3e} vs tol {float(tol[mask].max()):.3e}")
    return worst

"""Failure detection on the GPU without a fault: a wait that nothing satisfies runs into its
deadline, the kernel records the timeout and returns, the host reads CAST_ERR_DEVICE_TIMEOUT
from cast_check_device, and the context keeps working."""
import time

import numpy as np
import pytest
import torch

from tests.test_gpu_attention import _inputs, _rel_err
from tests.gpu_util import ATTN_REL_MAX, to_dev, to_host

import oracle.cast_oracle as O

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives(lib):
    lib.cast_check_device()                       # nothing pending
    t0 = time.perf_counter()
    lib.cast_selftest_bounded_wait(20_000_000)    # 20 ms deadline
    with pytest.raises(lib.CastError) as e:
        lib.cast_check_device()
    assert e.value.status == lib.ERR_DEVICE_TIMEOUT
    assert time.perf_counter() - t0 < 5.0
    lib.cast_check_device()                       # the record was cleared
    # the same context still runs the path correctly
    N, S, H, d, M, Bv, K = 2, 130, 2, 128, 3, 64, 2
    q, kc, vc, kh, vh = _inputs(9, N, S, H, d, M, Bv)
    idx = np.array([[[0, 2], [1, 2]]], dtype=np.int32)
    dk = (lambda x: to_dev(x, "bf16"))
    o = lib.cast_anchor_attention(dk(q), dk(kc), dk(vc), [1], dk(kh), dk(vh),
                                  torch.from_numpy(idx).cuda(), out_dtype=torch.float32)
    torch.cuda.synchronize()
    lib.cast_check_device()
    ref = O.routed_attention(q, kc, vc, kh, vh, [1], idx)
    assert _rel_err(to_host(o), ref.reshape(1, S, H * d)) <= ATTN_REL_MAX


def test_bounded_wait_limit_validation(lib):
    for bad in (0, 10, 3_000_000_000):
        with pytest.raises(lib.CastError) as e:
            lib.cast_selftest_bounded_wait(bad)
        assert e.value.status == lib.ERR_INVALID_ARG

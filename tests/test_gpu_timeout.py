"""Failure detection of the bounded device waits, without a GPU fault.

p4q_test_wait_timeout launches one warp whose mbarrier wait nothing ever
completes: the wait must give up after its limit, the kernel must return, the
next p4q_device_status must report P4Q_ERR_TIMEOUT once (reading clears it),
and the context must stay usable: an exact GEMM right after still matches the
oracle bit for bit."""
import ctypes
import time

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

P4Q_ERR_TIMEOUT = 6


def test_expired_wait_is_reported_and_the_context_survives(p4q, dev):
    stream = torch.cuda.current_stream()
    assert p4q.p4q_device_status() == 0
    t0 = time.perf_counter()
    assert p4q.lib().p4q_test_wait_timeout(2000, ctypes.c_void_p(stream.cuda_stream)) == 0
    assert p4q.p4q_device_status() == P4Q_ERR_TIMEOUT
    waited = time.perf_counter() - t0
    assert 0.0015 < waited < 1.0  # the 2 ms limit, not the 4 s default, ended the wait
    assert p4q.p4q_device_status() == 0  # reported once, then cleared

    rng = np.random.default_rng(11)
    a = rng.integers(-8, 8, size=(64, 256), dtype=np.int8)
    w = rng.integers(-8, 8, size=(128, 256), dtype=np.int8)
    Xq = torch.from_numpy(oracle.pack_codes(a)).to(dev)
    Wq = torch.from_numpy(oracle.pack_codes(w)).to(dev)
    acc = p4q.w4a4_gemm_s32(Xq, Wq)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    assert np.array_equal(acc.cpu().numpy(), oracle.gemm_s32(a, w))

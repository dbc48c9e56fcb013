"""The W4A4 linear at decode sizes (M <= 8 rows: the weight-streaming
kernel of the automatic dispatch) against the oracle: int32 accumulators
bit-exact, fp16 outputs within the linear tolerance."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _packed(rng, rows, K):
    return oracle.pack_codes(rng.integers(-8, 8, size=(rows, K), dtype=np.int8))


@pytest.mark.parametrize("M", [1, 2, 3, 4, 7, 8, 13, 16])
@pytest.mark.parametrize("N,K", [(11008, 4096), (4096, 11008), (264, 128), (8, 256), (13824, 5120)])
def test_gemv_s32_bit_exact(p4q, dev, M, N, K):
    rng = np.random.default_rng(M * 31 + N + K)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    acc = p4q.w4a4_gemm_s32(torch.from_numpy(a).to(dev), torch.from_numpy(w).to(dev))
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    assert np.array_equal(acc.cpu().numpy(), ref)


@pytest.mark.parametrize("M,N,K", [(1, 11008, 4096), (8, 4096, 11008), (5, 4096, 4096), (2, 256, 16384)])
def test_gemv_linear_fp16(p4q, dev, M, N, K):
    rng = np.random.default_rng(K + N + M)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    sa = (rng.random(M) * 0.5 + 0.01).astype(np.float32)
    sw = (rng.random(N) * 0.002 + 1e-4).astype(np.float32)
    Y = torch.empty((M, N), dtype=torch.float16, device=dev)
    p4q.p4q_w4a4_linear(torch.from_numpy(a).to(dev), torch.from_numpy(sa).to(dev), torch.from_numpy(w).to(dev),
                        torch.from_numpy(sw).to(dev), Y)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref = oracle.linear(oracle.unpack_codes(a), sa, oracle.unpack_codes(w), sw)
    # same epilogue as the oracle ((float)acc * s_a) * s_w in fp32, then fp16
    assert np.array_equal(Y.cpu().numpy(), ref.astype(np.float16))


def test_gemv_extreme_codes(p4q, dev):
    K = 16384
    pat = [0x77, 0x99, 0x88, 0x97, 0x00]
    a = np.stack([np.full(K // 2, p, np.uint8) for p in pat] * 2)[:8]
    w = np.stack([np.full(K // 2, p, np.uint8) for p in pat] * 60)[:296]
    acc = p4q.w4a4_gemm_s32(torch.from_numpy(a).to(dev), torch.from_numpy(w).to(dev))
    torch.cuda.synchronize()
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    assert np.array_equal(acc.cpu().numpy(), ref)

"""Pins for the oracle's W4A4 integer matmul and dequant (CPU only).

The linear follows App. B.3 (INT4 weights with one scale per output channel,
INT4 activations with one scale per token): acc = sum_k a[m,k] w[n,k] exactly,
y = (acc * s_a[m]) * s_w[n]. Pinned against numpy's int64 matmul, closed forms
for extreme codes, and float64 dequantization.
"""
import numpy as np
import pytest

import oracle


@pytest.mark.parametrize("M,N,K", [(1, 1, 2), (3, 5, 8), (17, 9, 130), (64, 48, 256)])
def test_gemm_matches_numpy_int64(M, N, K):
    rng = np.random.default_rng(M * 1000 + N)
    a = rng.integers(-8, 8, size=(M, K)).astype(np.int8)
    w = rng.integers(-8, 8, size=(N, K)).astype(np.int8)
    ref = a.astype(np.int64) @ w.astype(np.int64).T
    got = oracle.gemm_s32(a, w)
    assert got.dtype == np.int32 and np.array_equal(got.astype(np.int64), ref)


def test_gemm_extreme_codes_closed_form():
    K = 13824
    p7 = np.full((2, K), 7, np.int8)
    m7 = np.full((1, K), -7, np.int8)
    alt = np.tile(np.array([7, -7], np.int8), K // 2)[None]
    m8 = np.full((1, K), -8, np.int8)
    acc = oracle.gemm_s32(np.concatenate([p7, m7, alt, m8]), np.concatenate([p7[:1], m7, alt, m8]))
    assert acc[0, 0] == 49 * K and acc[0, 1] == -49 * K and acc[2, 1] == 49 * K
    assert acc[3, 2] == 49 * K and acc[0, 2] == 0
    assert acc[4, 3] == 64 * K and acc[4, 0] == -56 * K


def test_linear_matches_float64_dequant():
    rng = np.random.default_rng(3)
    M, N, K = 20, 30, 512
    a = rng.integers(-7, 8, size=(M, K)).astype(np.int8)
    w = rng.integers(-7, 8, size=(N, K)).astype(np.int8)
    sa = (rng.random(M) * 2 + 0.01).astype(np.float32)
    sw = (rng.random(N) * 0.01 + 1e-4).astype(np.float32)
    y = oracle.linear(a, sa, w, sw)
    ref = (a.astype(np.float64) @ w.astype(np.float64).T) * sa[:, None].astype(np.float64) \
        * sw[None, :].astype(np.float64)
    np.testing.assert_allclose(y, ref, rtol=3e-7, atol=1e-30)


def test_linear_of_quantized_fp_matmul_is_close():
    """End to end: quantize x and W, the W4A4 linear approximates x W^T (4-bit error)."""
    rng = np.random.default_rng(4)
    x = rng.standard_normal((16, 1024)).astype(np.float16)
    W = (rng.standard_normal((32, 1024)) * 0.02).astype(np.float16)
    ca, sa = oracle.quantize_rows(x)
    cw, sw = oracle.quantize_rows(W)
    y = oracle.linear(ca, sa, cw, sw)
    ref = x.astype(np.float64) @ W.astype(np.float64).T
    rel = np.linalg.norm(y - ref) / np.linalg.norm(ref)
    assert rel < 0.25

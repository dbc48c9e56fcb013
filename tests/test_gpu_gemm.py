"""GPU parity of the W4A4 integer GEMM (tcgen05, FP8 path) against the oracle:
int32 accumulators bit-exact; fp16 dequantized outputs within 1e-3 relative
(2e-3 absolute floor) of the oracle's fp32 dequant."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _packed(rng, rows, K):
    return rng.integers(0, 256, size=(rows, K // 2), dtype=np.uint8)  # any byte is a valid pair of codes


def _gemm(p4q, dev, a, w):
    acc = p4q.w4a4_gemm_s32(torch.from_numpy(a).to(dev), torch.from_numpy(w).to(dev))
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    return acc.cpu().numpy()


@pytest.fixture(params=[1, 2], ids=["single_cta", "cta_pair"])
def variant(request, p4q):
    p4q.p4q_set_gemm_variant(request.param)
    yield request.param
    p4q.p4q_set_gemm_variant(0)


@pytest.mark.parametrize("M,N,K", [(1, 8, 128), (128, 128, 128), (96, 4096, 4096), (200, 136, 256),
                                   (300, 1032, 384), (129, 1024, 1024), (64, 2048, 11008),
                                   (1100, 2056, 256), (2048, 4096, 512), (256, 256, 128), (257, 264, 256)])
def test_gemm_s32_bit_exact(p4q, dev, variant, M, N, K):
    rng = np.random.default_rng(M * 7 + N)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    got = _gemm(p4q, dev, a, w)
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    bad = np.argwhere(got != ref)
    assert bad.size == 0, f"{len(bad)} of {ref.size} differ, first {bad[:4].tolist()}"


@pytest.mark.parametrize("K", [13824, 16384])
def test_gemm_extreme_codes_exact(p4q, dev, variant, K):
    """Largest magnitudes: +7 x +7 (offset codes 15 x 15), -8 x -8, -8 x +7, and alternating signs."""
    pat = {"p7": 0x77, "m7": 0x99, "m8": 0x88, "alt": 0x97, "zero": 0x00}
    names = list(pat)
    a = np.stack([np.full(K // 2, pat[n], np.uint8) for n in names] * 26)[:128]
    w = np.stack([np.full(K // 2, pat[n], np.uint8) for n in names] * 52)[:256]
    got = _gemm(p4q, dev, a, w)
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    assert np.array_equal(got, ref)
    assert ref.max() == 64 * K


def test_gemm_zero_rows_is_noop(p4q, dev):
    a = torch.empty((0, 64), dtype=torch.uint8, device=dev)
    w = torch.zeros((8, 64), dtype=torch.uint8, device=dev)
    acc = torch.empty((0, 8), dtype=torch.int32, device=dev)
    p4q.p4q_w4a4_gemm_s32(a, w, acc)


@pytest.mark.parametrize("M,N,K", [(96, 4096, 4096), (257, 1032, 512), (33, 128, 13824), (2048, 4096, 1024),
                                   (300, 11008, 256), (512, 264, 128)])
def test_linear_fp16_within_tolerance(p4q, dev, variant, M, N, K):
    rng = np.random.default_rng(K + M)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    sa = (rng.random(M) * 0.5 + 0.01).astype(np.float32)
    sw = (rng.random(N) * 0.002 + 1e-4).astype(np.float32)
    Y = p4q.w4a4_linear(torch.from_numpy(a).to(dev), torch.from_numpy(sa).to(dev),
                        torch.from_numpy(w).to(dev), torch.from_numpy(sw).to(dev))
    torch.cuda.synchronize()
    y = Y.float().cpu().numpy()
    ref = oracle.linear(oracle.unpack_codes(a), sa, oracle.unpack_codes(w), sw)
    err = np.abs(y - ref)
    lim = np.maximum(1e-3 * np.abs(ref), 2e-3)
    assert np.all(err <= lim), f"max err {err.max()} at {np.unravel_index(np.argmax(err - lim), err.shape)}"


# ---------------------------------------------------------------- expanded-operand path (workspace entry points)
@pytest.fixture
def expanded(p4q):
    """Forces the expanded-operand path of the workspace entry points (also below 512 rows)."""
    p4q.p4q_set_gemm_variant(3)
    yield
    p4q.p4q_set_gemm_variant(0)


@pytest.mark.parametrize("M,N,K", [(1, 256, 128), (200, 264, 256), (256, 256, 128), (257, 264, 256),
                                   (600, 1032, 384), (2048, 4096, 512), (1100, 2056, 4096), (64, 2048, 11008)])
def test_expanded_gemm_s32_bit_exact(p4q, dev, expanded, M, N, K):
    rng = np.random.default_rng(M * 13 + N + 5)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    ws = p4q.linear_workspace(M, N, K, dev)
    acc = p4q.w4a4_gemm_s32_ws(torch.from_numpy(a).to(dev), torch.from_numpy(w).to(dev), ws)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    assert np.array_equal(acc.cpu().numpy(), ref)


@pytest.mark.parametrize("K", [13824, 16384])
def test_expanded_gemm_extreme_codes_exact(p4q, dev, expanded, K):
    pat = {"p7": 0x77, "m7": 0x99, "m8": 0x88, "alt": 0x97, "zero": 0x00}
    names = list(pat)
    a = np.stack([np.full(K // 2, pat[n], np.uint8) for n in names] * 26)[:128]
    w = np.stack([np.full(K // 2, pat[n], np.uint8) for n in names] * 52)[:256]
    ws = p4q.linear_workspace(128, 256, K, dev)
    acc = p4q.w4a4_gemm_s32_ws(torch.from_numpy(a).to(dev), torch.from_numpy(w).to(dev), ws)
    torch.cuda.synchronize()
    ref = oracle.gemm_s32(oracle.unpack_codes(a), oracle.unpack_codes(w))
    assert np.array_equal(acc.cpu().numpy(), ref)


@pytest.mark.parametrize("M,N,K", [(2048, 4096, 4096), (512, 264, 128), (1024, 13824, 5120), (700, 4096, 11008)])
def test_expanded_linear_fp16_within_tolerance(p4q, dev, M, N, K):
    """Automatic dispatch (M >= 512 takes the expanded path) through p4q_w4a4_linear_ws."""
    rng = np.random.default_rng(K + M + 1)
    a, w = _packed(rng, M, K), _packed(rng, N, K)
    sa = (rng.random(M) * 0.5 + 0.01).astype(np.float32)
    sw = (rng.random(N) * 0.002 + 1e-4).astype(np.float32)
    ws = p4q.linear_workspace(M, N, K, dev)
    Y = torch.empty((M, N), dtype=torch.float16, device=dev)
    p4q.p4q_w4a4_linear_ws(torch.from_numpy(a).to(dev), torch.from_numpy(sa).to(dev), torch.from_numpy(w).to(dev),
                           torch.from_numpy(sw).to(dev), Y, ws)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    y = Y.float().cpu().numpy()
    ref = oracle.linear(oracle.unpack_codes(a), sa, oracle.unpack_codes(w), sw)
    err = np.abs(y - ref)
    lim = np.maximum(1e-3 * np.abs(ref), 2e-3)
    assert np.all(err <= lim), f"max err {err.max()}"


def test_expanded_linear_rejects_a_short_workspace(p4q, dev):
    Xq = torch.zeros((1024, 2048), dtype=torch.uint8, device=dev)
    Wq = torch.zeros((512, 2048), dtype=torch.uint8, device=dev)
    s = torch.ones((1024,), dtype=torch.float32, device=dev)
    Y = torch.empty((1024, 512), dtype=torch.float16, device=dev)
    short = torch.empty((1024,), dtype=torch.uint8, device=dev)
    with pytest.raises(p4q.P4QError):
        p4q.p4q_w4a4_linear_ws(Xq, s, Wq, s[:512], Y, short)


def test_expand_codes_layout_and_sums(p4q, dev):
    """One byte u = v + 8 per code; per packed 32-bit word its four low-nibble
    codes, then its four high-nibble codes; sum_u per row."""
    rng = np.random.default_rng(3)
    q = _packed(rng, 37, 384)
    u, s = p4q.expand_codes(torch.from_numpy(q).to(dev))
    torch.cuda.synchronize()
    v = oracle.unpack_codes(q).astype(np.int32) + 8          # [rows, K] natural order
    w = v.reshape(37, -1, 4, 2)                              # [rows, word, byte, (lo, hi)]
    expect = np.concatenate([w[..., 0], w[..., 1]], axis=2).reshape(37, -1)
    assert np.array_equal(u.cpu().numpy().astype(np.int32), expect)
    assert np.array_equal(s.cpu().numpy(), v.sum(axis=1))


def test_linear_expanded_matches_linear(p4q, dev):
    rng = np.random.default_rng(4)
    M, N, K = 300, 512, 1024
    a, w = torch.from_numpy(_packed(rng, M, K)).to(dev), torch.from_numpy(_packed(rng, N, K)).to(dev)
    sa = torch.rand(M, device=dev) * 0.3 + 0.01
    sw = torch.rand(N, device=dev) * 0.002 + 1e-4
    ref = p4q.w4a4_linear(a, sa, w, sw)
    Xu, sX = p4q.expand_codes(a)
    Wu, sW = p4q.expand_codes(w)
    Y = torch.empty((M, N), dtype=torch.float16, device=dev)
    p4q.p4q_w4a4_linear_expanded(Xu, sX, sa, Wu, sW, sw, Y)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    assert torch.equal(Y.view(torch.int16), ref.view(torch.int16))

"""GPU parity of SwiGLU -> per-token INT4 (the input of down_proj) against the
float64 oracle (silu with the C library's exp): scales within 1e-6, codes
identical except where the float64 quotient h / s lies within the kernel's
error bound of a .5 boundary (reading R12: the kernel's fp32 quotient is
within 5.7e-6 and the oracle's within 1.7e-6 of the exact one; the band is
1e-5), expanded codes and row sums
consistent with the packed ones."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _run(p4q, dev, G, U, expanded=True):
    M, K = G.shape
    Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
    s = torch.empty((M,), dtype=torch.float32, device=dev)
    Xu = torch.empty((M, K), dtype=torch.uint8, device=dev) if expanded else None
    su = torch.empty((M,), dtype=torch.int32, device=dev) if expanded else None
    p4q.p4q_swiglu_quant_expanded(G, U, Xq, s, Xu, su)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    return Xq.cpu().numpy(), s.cpu().numpy(), (None if Xu is None else Xu.cpu().numpy()), \
        (None if su is None else su.cpu().numpy())


FLT_MIN = float(np.finfo(np.float32).tiny)
BAND = 1e-5           # codes are compared where the float64 quotient is this far from a .5 boundary
SATURATE = -88.72284  # below this gate the kernel's exponential of -g is inf: silu(g) = 0


def _check(p4q, dev, g, u, expanded=True, G=None, U=None):
    G = torch.from_numpy(g).to(dev) if G is None else G
    U = torch.from_numpy(u).to(dev) if U is None else U
    q, s, xu, su = _run(p4q, dev, G, U, expanded)
    got = oracle.unpack_codes(q)
    c, sr = oracle.swiglu_quantize_rows(g, u)
    gd, ud = g.astype(np.float64), u.astype(np.float64)
    with np.errstate(over="ignore"):  # exp(-g) = inf for very negative gates: silu = 0
        h = gd / (1.0 + np.exp(-gd)) * ud
    a = np.abs(h).max(axis=1)
    # rows whose values lie below the fp32 normal range, or whose every gate
    # saturates the kernel's exponential, come back as zero rows
    tiny = (a < FLT_MIN) | np.all(gd < SATURATE, axis=1)
    assert not got[tiny].any() and not s[tiny].any(), "a flushed row is not zero"
    ok = ~tiny
    assert np.all(np.abs(s[ok].astype(np.float64) / sr[ok] - 1.0) <= 1e-6), "scales differ"
    qq = h[ok] / (a[ok] / 7.0)[:, None]
    near = np.abs(np.abs(qq - np.floor(qq)) - 0.5) < BAND
    g_ok, c_ok = got[ok], c[ok]
    bad = np.argwhere((g_ok != c_ok) & ~near)
    assert bad.size == 0, f"{len(bad)} codes differ away from a .5 boundary, first at {bad[:3].tolist()}"
    assert np.all(np.abs(g_ok[near] - qq[near]) <= 0.5 + BAND)
    if expanded:
        # per 32-bit word of packed codes: its four even-index codes, then its four odd ones, + 8
        K = g.shape[1]
        w = (got.astype(np.int16) + 8).reshape(-1, K // 8, 8)
        want = np.concatenate([w[..., 0::2], w[..., 1::2]], axis=-1).reshape(-1, K).astype(np.uint8)
        assert np.array_equal(xu, want)
        assert np.array_equal(su, want.astype(np.int64).sum(1))


@pytest.mark.parametrize("M,K", [(1, 16), (7, 128), (33, 4096), (64, 11008), (5, 16384), (300, 13824)])
def test_swiglu_quant_matches_oracle(p4q, dev, M, K):
    rng = np.random.default_rng(M + K)
    g = (rng.standard_normal((M, K)) * 3).astype(np.float16)
    u = (rng.standard_normal((M, K)) * 2).astype(np.float16)
    _check(p4q, dev, g, u)


def test_swiglu_quant_extremes(p4q, dev):
    """Gates past the kernel exponential's cuts (inf and 0 branches), fp16
    extremes, zero rows, rows where every gate is very negative (zero rows)."""
    rng = np.random.default_rng(9)
    K = 1024
    g = (rng.standard_normal((8, K)) * 40).astype(np.float16)
    u = (rng.standard_normal((8, K)) * 3).astype(np.float16)
    g[0, :8] = [65504, -65504, 88.75, -88.75, 87.0, -87.0, 0.0, -0.0]
    g[1] = -100.0
    u[2] = 0.0
    g[3] = 0.0
    u[4, :4] = [65504, -65504, 1e-7, -1e-7]
    _check(p4q, dev, g, u)


def test_swiglu_quant_column_blocks_without_expanded(p4q, dev):
    """gate and up as column blocks of one fused output (row pitch > Kin), packed codes only."""
    rng = np.random.default_rng(3)
    M, K, W = 48, 2048, 2 * 2048 + 512
    Y = (rng.standard_normal((M, W)) * 2).astype(np.float16)
    Yd = torch.from_numpy(Y).to(dev)
    g, u = Y[:, 512:512 + K], Y[:, 512 + K:512 + 2 * K]
    _check(p4q, dev, np.ascontiguousarray(g), np.ascontiguousarray(u), expanded=False,
           G=Yd[:, 512:512 + K], U=Yd[:, 512 + K:512 + 2 * K])

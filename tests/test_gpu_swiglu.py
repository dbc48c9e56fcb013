"""GPU parity of SwiGLU -> per-token INT4 (the input of down_proj) against the
oracle: codes, scale bits, expanded codes and their row sums bit-exact."""
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


def _check(p4q, dev, g, u, expanded=True, G=None, U=None):
    G = torch.from_numpy(g).to(dev) if G is None else G
    U = torch.from_numpy(u).to(dev) if U is None else U
    q, s, xu, su = _run(p4q, dev, G, U, expanded)
    c, sr = oracle.swiglu_quantize_rows(g, u)
    assert np.array_equal(s.view(np.uint32), sr.view(np.uint32)), "scale bits differ"
    got = oracle.unpack_codes(q)
    bad = np.argwhere(got != c)
    assert bad.size == 0, f"{len(bad)} codes differ, first at {bad[:3].tolist()}"
    if expanded:
        # per 32-bit word of packed codes: its four even-index codes, then its four odd ones, + 8
        K = g.shape[1]
        w = (c.astype(np.int16) + 8).reshape(-1, K // 8, 8)
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
    """Gates past exp32's cuts (inf and 0 branches), fp16 extremes, zero rows,
    rows where every gate is very negative (h = -0 * u)."""
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

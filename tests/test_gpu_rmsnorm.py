"""GPU parity of RMSNorm -> per-token INT4 (the input of the decoder's
quantized linears) against the oracle: codes, scale bits, expanded codes and
their row sums bit-exact."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _run(p4q, dev, X, w, eps, expanded=True):
    M, K = X.shape
    Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
    s = torch.empty((M,), dtype=torch.float32, device=dev)
    Xu = torch.empty((M, K), dtype=torch.uint8, device=dev) if expanded else None
    su = torch.empty((M,), dtype=torch.int32, device=dev) if expanded else None
    p4q.p4q_rmsnorm_quant_expanded(X, w, eps, Xq, s, Xu, su)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    return Xq.cpu().numpy(), s.cpu().numpy(), (None if Xu is None else Xu.cpu().numpy()), \
        (None if su is None else su.cpu().numpy())


def _check(p4q, dev, x, w, eps, expanded=True, X=None):
    X = torch.from_numpy(x).to(dev) if X is None else X
    q, s, xu, su = _run(p4q, dev, X, torch.from_numpy(w).to(dev), eps, expanded)
    c, sr = oracle.rmsnorm_quantize_rows(x, w, eps)
    assert np.array_equal(s.view(np.uint32), sr.view(np.uint32)), "scale bits differ"
    got = oracle.unpack_codes(q)
    bad = np.argwhere(got != c)
    assert bad.size == 0, f"{len(bad)} codes differ, first at {bad[:3].tolist()}"
    if expanded:
        # per 32-bit word of packed codes: its four even-index codes, then its four odd ones, + 8
        K = x.shape[1]
        v = (c.astype(np.int16) + 8).reshape(-1, K // 8, 8)
        want = np.concatenate([v[..., 0::2], v[..., 1::2]], axis=-1).reshape(-1, K).astype(np.uint8)
        assert np.array_equal(xu, want)
        assert np.array_equal(su, want.astype(np.int64).sum(1))


@pytest.mark.parametrize("M,K,eps", [(1, 16, 1e-6), (7, 128, 1e-5), (33, 4096, 1e-6), (64, 5120, 1e-5),
                                     (5, 16384, 1e-6), (300, 4096, 0.5)])
def test_rmsnorm_quant_matches_oracle(p4q, dev, M, K, eps):
    rng = np.random.default_rng(M + K)
    x = (rng.standard_normal((M, K)) * rng.uniform(0.01, 30, (M, 1))).astype(np.float16)
    w = (1.0 + 0.5 * rng.standard_normal(K)).astype(np.float16)
    _check(p4q, dev, x, w, eps)


def test_rmsnorm_quant_extremes(p4q, dev):
    """Rows of fp16 subnormals only (the sum below 2^64 units), of the largest
    values (above it), of both (the sticky bit), the tie of the rounded sum,
    zero rows with and without eps, zero and negative gains."""
    rng = np.random.default_rng(5)
    K = 1024
    x = (rng.standard_normal((10, K)) * 3).astype(np.float16)
    x[0] = (rng.integers(-1023, 1024, K) * 2.0 ** -24).astype(np.float16)           # subnormals
    x[1] = (rng.choice([-1, 1], K) * rng.uniform(30000, 65504, K)).astype(np.float16)
    x[2, ::2] = 65504.0
    x[2, 1::2] = np.float16(2.0 ** -24)
    x[3] = 0.0
    x[4, :] = 0.0
    x[4, :4] = [2.0 ** -12, 2.0 ** -24, 2.0 ** -24, 2.0 ** -24]                    # 2^24 + 3 units
    x[5, :] = np.float16(-2.0 ** -24)
    w = (rng.uniform(0.25, 3.0, K) * rng.choice([-1, 1], K)).astype(np.float16)
    w[:16] = 0.0
    for eps in (0.0, 1e-6):
        _check(p4q, dev, x, w, eps)


def test_rmsnorm_quant_row_pitch_without_expanded(p4q, dev):
    """X as a column block of a wider matrix (row pitch > Kin), packed codes only."""
    rng = np.random.default_rng(3)
    M, K, W = 48, 2048, 4096
    Y = (rng.standard_normal((M, W)) * 2).astype(np.float16)
    Yd = torch.from_numpy(Y).to(dev)
    w = (1.0 + 0.1 * rng.standard_normal(K)).astype(np.float16)
    _check(p4q, dev, np.ascontiguousarray(Y[:, 1024:1024 + K]), w, 1e-6, expanded=False, X=Yd[:, 1024:1024 + K])

"""Pins of the oracle's pruning-aware calibration data path: Eq. 5's block
objective (per-sample squared Frobenius distance over m_n d, then the batch
mean) and Eq. 9's Top-K replacement ratio (App. A), against closed forms,
exact sums and brute-force ranking."""
import math

import numpy as np

import oracle


def test_block_mse_closed_forms():
    rng = np.random.default_rng(0)
    Y = rng.standard_normal((10, 6)).astype(np.float32)
    off = [0, 4, 10]
    e, L = oracle.block_mse(Y, Y, off)
    assert np.array_equal(e, [0.0, 0.0]) and L == 0.0
    # a constant difference c in sample 0 and 2c in sample 1: e = c^2 and 4 c^2
    D = Y.copy()
    D[:4] += 0.5
    D[4:] -= 1.0
    e, L = oracle.block_mse(D, Y, off)
    assert np.allclose(e, [0.25, 1.0], rtol=1e-6) and math.isclose(L, 0.625, rel_tol=1e-6)


def test_block_mse_normalises_per_sample():
    # one differing element: its square divided by that sample's m_n d only
    Yf = np.zeros((7, 4), np.float32)
    Yq = Yf.copy()
    Yq[5, 2] = 3.0
    e, L = oracle.block_mse(Yq, Yf, [0, 2, 7])
    assert e.tolist() == [0.0, 9.0 / (5 * 4)] and L == 9.0 / 20 / 2


def test_block_mse_against_exact_sums():
    rng = np.random.default_rng(1)
    off = np.array([0, 256, 256 + 200, 256 + 200 + 320])
    Yq = rng.standard_normal((off[-1], 64)).astype(np.float16).astype(np.float32)
    Yf = (Yq + 0.01 * rng.standard_normal(Yq.shape)).astype(np.float16).astype(np.float32)
    e, L = oracle.block_mse(Yq, Yf, off)
    for n in range(3):
        d = (Yq[off[n]:off[n + 1]].astype(np.float64) - Yf[off[n]:off[n + 1]]).ravel()
        want = math.fsum((d * d).tolist()) / (d.size)
        assert math.isclose(e[n], want, rel_tol=1e-12)
    assert math.isclose(L, e.mean(), rel_tol=1e-15)


def _brute_topk(s, K):
    order = sorted(range(len(s)), key=lambda i: (-float(s[i]), i))
    return set(order[:K])


def test_replacement_ratio_brute_force():
    rng = np.random.default_rng(2)
    B, N = 6, 300
    s_ref = rng.standard_normal((B, N)).astype(np.float32)
    s_alt = (s_ref + 0.3 * rng.standard_normal((B, N))).astype(np.float32)
    s_alt[0, ::7] = s_alt[0, 0]  # ties, resolved to the lower index
    for K in (1, 33, 150, 300):
        inter, rho = oracle.topk_replacement(s_ref, s_alt, K)
        for b in range(B):
            c = len(_brute_topk(s_ref[b], K) & _brute_topk(s_alt[b], K))
            assert inter[b] == c
            assert rho[b] == np.float32(1.0) - np.float32(c) / np.float32(K)


def test_replacement_ratio_extremes():
    s = np.arange(100, dtype=np.float32)[None]
    inter, rho = oracle.topk_replacement(s, s, 20)
    assert inter[0] == 20 and rho[0] == 0.0
    inter, rho = oracle.topk_replacement(s, -s, 20)       # reversed ranking, 2K <= N: disjoint sets
    assert inter[0] == 0 and rho[0] == 1.0
    inter, rho = oracle.topk_replacement(s, -s, 100)      # K = N keeps everything
    assert inter[0] == 100 and rho[0] == 0.0
    flat = np.zeros((1, 10), np.float32)                  # all tied: the first K indices on both sides
    inter, _ = oracle.topk_replacement(flat, flat, 4)
    assert inter[0] == 4
    inter, _ = oracle.topk_replacement(flat, np.arange(10, dtype=np.float32)[None], 4)
    assert inter[0] == 0                                   # {0,1,2,3} against {6,7,8,9}

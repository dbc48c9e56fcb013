"""Pins of the oracle's causal attention on the pruned sequence (App. B:
FP16 key/value caches; softmax(q k^T / sqrt(d_h)) over positions 0..i):
closed forms, invariants and special cases independent of its loops."""
import math

import numpy as np

import oracle


def _rand(B, m, H, Hkv, dh, seed, scale=1.0):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal((B * m, H * dh)) * scale).astype(np.float16)
    k = (rng.standard_normal((B * m, Hkv * dh)) * scale).astype(np.float16)
    v = rng.standard_normal((B * m, Hkv * dh)).astype(np.float16)
    return q, k, v


def test_first_position_returns_its_value():
    q, k, v = _rand(3, 5, 2, 2, 8, seed=0)
    o = oracle.causal_attention(q, k, v, 3, 5, 2, 2, 8)
    for b in range(3):
        assert np.array_equal(o[b * 5], v[b * 5].astype(np.float64))


def test_two_positions_by_hand():
    # dh = 4, one head: q_1 = [1, 1, 0, 0], k_0 = [2, 0, 0, 0], k_1 = [0, 0, 2, 0]
    # logits 2 / 2 = 1 and 0: p_0 = 1 / (1 + e^-1)
    q = np.array([[0, 0, 0, 0], [1, 1, 0, 0]], np.float16)
    k = np.array([[2, 0, 0, 0], [0, 0, 2, 0]], np.float16)
    v = np.array([[1, 2, 3, 4], [-1, 0, 1, 0]], np.float16)
    o = oracle.causal_attention(q, k, v, 1, 2, 1, 1, 4)
    p0 = 1.0 / (1.0 + math.exp(-1.0))
    want = p0 * np.array([1, 2, 3, 4]) + (1 - p0) * np.array([-1, 0, 1, 0])
    assert np.allclose(o[1], want, rtol=0, atol=1e-15)
    assert np.array_equal(o[0], [1, 2, 3, 4])


def test_equal_keys_average_the_prefix():
    B, m, dh = 2, 9, 16
    q, _, v = _rand(B, m, 1, 1, dh, seed=1)
    key = np.random.default_rng(2).standard_normal(dh).astype(np.float16)
    k = np.tile(key, (B * m, 1))
    o = oracle.causal_attention(q, k, v, B, m, 1, 1, dh)
    vv = v.astype(np.float64).reshape(B, m, dh)
    want = np.cumsum(vv, axis=1) / np.arange(1, m + 1)[None, :, None]
    assert np.allclose(o.reshape(B, m, dh), want, rtol=0, atol=1e-14)


def test_future_positions_do_not_matter():
    B, m, H, dh = 1, 12, 2, 8
    q, k, v = _rand(B, m, H, H, dh, seed=3)
    o = oracle.causal_attention(q, k, v, B, m, H, H, dh)
    k2, v2 = k.copy(), v.copy()
    k2[7:] = np.random.default_rng(4).standard_normal(k2[7:].shape).astype(np.float16)
    v2[7:] = 0
    o2 = oracle.causal_attention(q, k2, v2, B, m, H, H, dh)
    assert np.array_equal(o[:7], o2[:7]) and not np.allclose(o[7:], o2[7:])


def test_samples_are_independent():
    q, k, v = _rand(3, 6, 1, 1, 8, seed=5)
    o = oracle.causal_attention(q, k, v, 3, 6, 1, 1, 8)
    o_mid = oracle.causal_attention(q[6:12], k[6:12], v[6:12], 1, 6, 1, 1, 8)
    assert np.array_equal(o[6:12], o_mid)


def test_dominant_key_selects_its_value():
    # q_i = 8 e_i and k_j = 8 e_j: logit 64 / sqrt(16) = 16 on the diagonal, 0 elsewhere
    m, dh = 10, 16
    eye = (8 * np.eye(m, dh)).astype(np.float16)
    v = np.random.default_rng(6).standard_normal((m, dh)).astype(np.float16)
    o = oracle.causal_attention(eye, eye, v, 1, m, 1, 1, dh)
    for i in range(m):
        w = np.full(i + 1, 1.0)
        w[i] = math.exp(16.0)
        want = (w[:, None] * v[:i + 1].astype(np.float64)).sum(0) / w.sum()
        assert np.allclose(o[i], want, rtol=1e-13, atol=1e-15)


def test_output_is_linear_in_values_and_a_convex_combination():
    B, m, H, dh = 2, 7, 2, 8
    q, k, v = _rand(B, m, H, H, dh, seed=7, scale=2.0)
    o = oracle.causal_attention(q, k, v, B, m, H, H, dh)
    o2 = oracle.causal_attention(q, k, (2 * v.astype(np.float32)).astype(np.float16), B, m, H, H, dh)
    assert np.allclose(o2, 2 * o, rtol=1e-14, atol=0)
    vv = v.astype(np.float64).reshape(B, m, H, dh)
    oo = o.reshape(B, m, H, dh)
    for i in range(m):
        lo, hi = vv[:, :i + 1].min(axis=1), vv[:, :i + 1].max(axis=1)
        assert np.all(oo[:, i] >= lo - 1e-12) and np.all(oo[:, i] <= hi + 1e-12)


def test_grouped_heads_share_their_key_value_head():
    B, m, H, Hkv, dh = 1, 8, 4, 2, 8
    q, k, v = _rand(B, m, H, Hkv, dh, seed=8)
    o = oracle.causal_attention(q, k, v, B, m, H, Hkv, dh)
    for h in range(H):
        hk = h // 2
        oh = oracle.causal_attention(q[:, h * dh:(h + 1) * dh], k[:, hk * dh:(hk + 1) * dh],
                                     v[:, hk * dh:(hk + 1) * dh], B, m, 1, 1, dh)
        assert np.array_equal(o[:, h * dh:(h + 1) * dh], oh)


def test_shifting_every_key_keeps_the_weights():
    # adding the same vector to every key shifts all logits of a row by q . c:
    # the weights do not change (up to rounding of the shifted fp16 keys)
    m, dh = 6, 8
    q, k, v = _rand(1, m, 1, 1, dh, seed=9)
    c = np.random.default_rng(10).standard_normal(dh).astype(np.float16)
    o = oracle.causal_attention(q, k, v, 1, m, 1, 1, dh)
    o2 = oracle.causal_attention(q, (k.astype(np.float32) + c.astype(np.float32)).astype(np.float16), v, 1, m, 1, 1,
                                 dh)
    assert np.allclose(o2, o, atol=2e-2)

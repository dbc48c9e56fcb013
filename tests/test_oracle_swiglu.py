"""Pins of the oracle's SwiGLU -> per-token 4-bit quantizer (the input of
down_proj; App. A quantizes every linear's input per token) and of its own
fp32 exponential: float64 mathematics, closed forms and special cases."""
import math

import numpy as np

import oracle


def test_exp32_is_within_one_ulp_of_exp():
    x = np.linspace(-87.0, 88.7, 400001).astype(np.float32)
    y = oracle.exp32(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(y - ref) / ulp) < 1.0


def test_exp32_exact_points_and_range():
    assert oracle.exp32(np.zeros(1))[0] == 1.0
    # at the fp32 roundings of k ln 2 (whose exact exponentials are close to 2^k)
    k = np.arange(-125, 127)
    x = (k * math.log(2)).astype(np.float32)
    y = oracle.exp32(x).astype(np.float64)
    assert np.all(np.abs(y / np.exp(x.astype(np.float64)) - 1.0) < 1.2e-7)
    assert np.all(np.abs(y / np.exp2(k.astype(np.float64)) - 1.0) < 1e-5)
    assert np.isinf(oracle.exp32(np.array([89.0]))[0])
    assert oracle.exp32(np.array([-87.01]))[0] == 0.0
    assert oracle.exp32(np.array([-87.0]))[0] > np.finfo(np.float32).tiny  # normal down to the cut


def test_swiglu_worked_row():
    # h = silu(g) * 1 = g / (1 + e^-g): [0.7310586, -0.2689414, 1.7615942, 0]
    g = np.array([[1.0, -1.0, 2.0, 0.0]], np.float32)
    u = np.ones_like(g)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    h = g.astype(np.float64) / (1.0 + np.exp(-g.astype(np.float64)))
    assert abs(scale[0] - h.max() / 7.0) < 1e-7
    assert codes.tolist() == [[3, -1, 7, 0]]   # h / s = [2.905, -1.069, 7, 0]


def test_large_gates_reduce_to_the_product():
    # g >= 17: exp(-g) < 2^-24, so 1 + exp(-g) rounds to 1 and silu(g) = g
    rng = np.random.default_rng(0)
    g = (rng.random((8, 256)) * 100 + 17).astype(np.float32)
    u = rng.standard_normal((8, 256)).astype(np.float32)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    c2, s2 = oracle.quantize_rows(g * u)
    assert np.array_equal(codes, c2) and np.array_equal(scale.view(np.uint32), s2.view(np.uint32))


def test_very_negative_gates_give_zero_rows():
    g = np.full((3, 64), -100.0, np.float32)
    u = np.random.default_rng(1).standard_normal((3, 64)).astype(np.float32)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    assert not codes.any() and not scale.any()


def test_swiglu_against_float64():
    rng = np.random.default_rng(2)
    g = (rng.standard_normal((64, 512)) * 3).astype(np.float16).astype(np.float32)
    u = (rng.standard_normal((64, 512)) * 2).astype(np.float16).astype(np.float32)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    h = g.astype(np.float64) / (1.0 + np.exp(-g.astype(np.float64))) * u
    a = np.abs(h).max(axis=1)
    assert np.all(np.abs(scale / (a / 7.0) - 1.0) < 1e-6)
    q = h / (a / 7.0)[:, None]
    near = np.abs(np.abs(q - np.floor(q)) - 0.5) < 1e-4   # within rounding distance of a .5 boundary
    want = np.clip(np.rint(q), -8, 7)
    assert np.array_equal(codes[~near], want[~near].astype(np.int8))
    assert np.all(np.abs(codes[near] - q[near]) <= 0.5 + 1e-4)

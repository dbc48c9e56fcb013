"""Pins of the oracle's SwiGLU -> per-token 4-bit quantizer (the input of
down_proj; App. A quantizes every linear's input per token): a hand-worked
row, closed forms and special cases, and float64 mathematics."""
import numpy as np

import oracle


def test_swiglu_worked_row():
    # h = silu(g) * 1 = g / (1 + e^-g): [0.7310586, -0.2689414, 1.7615942, 0]
    g = np.array([[1.0, -1.0, 2.0, 0.0]], np.float32)
    u = np.ones_like(g)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    h = g.astype(np.float64) / (1.0 + np.exp(-g.astype(np.float64)))
    assert abs(scale[0] - h.max() / 7.0) < 1e-7
    assert codes.tolist() == [[3, -1, 7, 0]]   # h / s = [2.905, -1.069, 7, 0]


def test_swiglu_is_silu_times_up_rounded_once():
    # silu(0) = 0, silu(ln 3) = ln 3 * 3/4 exactly in the reals; odd-symmetric part:
    # silu(g) - silu(-g) = g
    g = np.array([[0.0, np.log(3.0), 2.5, -2.5]], np.float32)
    u = np.array([[5.0, 4.0, 1.0, 1.0]], np.float32)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    gd = g.astype(np.float64)
    h = np.float32(gd / (1.0 + np.exp(-gd)) * u)
    assert abs(float(h[0, 1]) - np.log(3.0) * 0.75 * 4.0) < 1e-6
    assert abs(float(h[0, 2]) - float(h[0, 3]) - 2.5) < 1e-6
    c2, s2 = oracle.quantize_rows(h)
    assert np.array_equal(codes, c2) and np.array_equal(scale.view(np.uint32), s2.view(np.uint32))


def test_large_gates_reduce_to_the_product():
    # g >= 40: exp(-g) < 2^-57, so silu(g) * u rounds to the (exact) fp32 product g * u
    rng = np.random.default_rng(0)
    g = (rng.random((8, 256)) * 100 + 40).astype(np.float16).astype(np.float32)
    u = rng.standard_normal((8, 256)).astype(np.float16).astype(np.float32)
    codes, scale = oracle.swiglu_quantize_rows(g, u)
    c2, s2 = oracle.quantize_rows(g * u)
    assert np.array_equal(codes, c2) and np.array_equal(scale.view(np.uint32), s2.view(np.uint32))


def test_very_negative_gates_give_zero_rows():
    # g <= -120: |silu(g) * u| < 2^-149 for |u| < 4, below the smallest fp32 magnitude
    g = np.full((3, 64), -120.0, np.float32)
    u = np.clip(np.random.default_rng(1).standard_normal((3, 64)), -3.9, 3.9).astype(np.float32)
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
    near = np.abs(np.abs(q - np.floor(q)) - 0.5) < 1e-5   # within rounding distance of a .5 boundary
    want = np.clip(np.rint(q), -8, 7)
    assert np.array_equal(codes[~near], want[~near].astype(np.int8))
    assert np.all(np.abs(codes[near] - q[near]) <= 0.5 + 1e-5)


def test_planted_fp32_exponential_is_detected():
    """An oracle built on a cruder exponential (expf evaluated as 2^(x log2 e)
    with the product rounded to fp32 first) differs from the float64 one on a
    sweep of gates: the pins above would see it."""
    g = np.linspace(-20.0, 20.0, 4001).astype(np.float32)
    u = np.ones_like(g)
    h64 = np.float32(g.astype(np.float64) / (1.0 + np.exp(-g.astype(np.float64))))
    crude = g / (np.float32(1.0) + np.exp2(np.float32(-g * np.float32(1.4426950408889634))))
    codes, _ = oracle.swiglu_quantize_rows(g[None, :], u[None, :])
    c64, _ = oracle.quantize_rows(h64[None, :])
    assert np.array_equal(codes, c64)
    assert not np.array_equal(h64, crude.astype(np.float32))

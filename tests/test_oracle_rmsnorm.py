"""Pins of the oracle's RMSNorm -> per-token 4-bit quantizer (the decoder's
input norms feed the quantized linears; App. A quantizes every linear's input
per token): exact rounding of the sum of squares, a hand-worked row, float64
mathematics, scale invariance and symmetry."""
import math

import numpy as np
import pytest

import oracle


def _f16(a):
    return np.asarray(a, np.float64).astype(np.float16)


def test_sum_of_squares_rounds_once_to_nearest_even():
    # 2^24 + 3 units of 2^-48: halfway between 2^24 + 2 and 2^24 + 4, the even
    # significand wins (a truncating or twice-rounding sum gives 2^24 + 2)
    x = _f16([2.0 ** -12, 2.0 ** -24, 2.0 ** -24, 2.0 ** -24])
    want = np.float32(float(2 ** 24 + 3)) * np.float32(2.0 ** -48)
    assert oracle.sumsq32(x) == want == np.float32(2 ** 24 + 4) * np.float32(2.0 ** -48)
    # 2^24 + 1 units: halfway, down to the even 2^24
    assert oracle.sumsq32(_f16([2.0 ** -12, 2.0 ** -24])) == np.float32(2.0 ** -24)


def test_sum_of_squares_is_exact_over_wide_ranges():
    rng = np.random.default_rng(0)
    for n in (1, 7, 4096, 16384):
        mag = 2.0 ** rng.integers(-24, 15, n)  # subnormals up to large normals
        x = _f16(mag * rng.uniform(0.5, 1.0, n) * rng.choice([-1, 1], n))
        exact = math.fsum((x.astype(np.float64) ** 2).tolist())  # squares of fp16 are exact in fp64
        assert oracle.sumsq32(x) == np.float32(exact)


def test_non_fp16_input_is_rejected():
    with pytest.raises(ValueError):
        oracle.sumsq32(np.array([0.1], np.float32))
    with pytest.raises(ValueError):
        oracle.rmsnorm_rows(np.array([[0.1, 1.0]], np.float32), np.ones(2, np.float16), 1e-6)


def test_worked_row():
    # x = [3, 4]: mean square 12.5, 1 / sqrt(12.5) = 0.28284271; x * r =
    # [0.84852814, 1.13137085] -> fp16 [0.8486328125, 1.1318359375]
    y = oracle.rmsnorm_rows(_f16([[3, 4]]), _f16([1, 1]), 0.0)
    assert y.tolist() == [[0.8486328125, 1.1318359375]]
    codes, scale = oracle.rmsnorm_quantize_rows(_f16([[3, 4]]), _f16([1, 1]), 0.0)
    assert codes.tolist() == [[5, 7]]  # y / (1.1318359375 / 7) = [5.2486, 7]
    assert scale[0] == np.float32(np.float32(1.1318359375) / np.float32(7))


@pytest.mark.parametrize("eps", [1e-6, 0.5])
def test_against_float64(eps):
    rng = np.random.default_rng(1)
    rows, d = 32, 1024
    x = _f16(rng.standard_normal((rows, d)) * rng.uniform(0.05, 20, (rows, 1)))
    w = _f16(1.0 + 0.3 * rng.standard_normal(d))
    y = oracle.rmsnorm_rows(x, w, eps).astype(np.float64)
    x64, w64 = x.astype(np.float64), w.astype(np.float64)
    t = (x64 / np.sqrt((x64 ** 2).mean(axis=1, keepdims=True) + eps)).astype(np.float16).astype(np.float64)
    want = (t * w64).astype(np.float16).astype(np.float64)
    ulp = np.spacing(np.abs(want).astype(np.float16)).astype(np.float64)
    assert np.all(np.abs(y - want) <= 2 * ulp)     # double rounding near fp16 ties may move one step per cast
    assert np.mean(y == want) > 0.999
    codes, scale = oracle.rmsnorm_quantize_rows(x, w, eps)
    a = np.abs(y).max(axis=1)
    assert np.all(np.abs(scale / (a / 7.0) - 1.0) < 1e-6)
    q = y / (a / 7.0)[:, None]
    near = np.abs(np.abs(q - np.floor(q)) - 0.5) < 1e-4
    assert np.array_equal(codes[~near], np.clip(np.rint(q), -8, 7)[~near].astype(np.int8))


def test_power_of_two_scaling_changes_nothing():
    # eps = 0: x * 2^j scales the exact sum by 4^j, the mean square, root and
    # reciprocal by exact powers of two, so y and the codes are unchanged
    rng = np.random.default_rng(2)
    x = _f16(rng.standard_normal((8, 512)) * 4)
    w = _f16(rng.uniform(0.5, 2.0, 512))
    c0, s0 = oracle.rmsnorm_quantize_rows(x, w, 0.0)
    for j in (-3, 1, 4):
        cj, sj = oracle.rmsnorm_quantize_rows(x * np.float16(2.0 ** j), w, 0.0)
        assert np.array_equal(cj, c0) and np.array_equal(sj.view(np.uint32), s0.view(np.uint32))


def test_negated_gain_negates_the_codes():
    rng = np.random.default_rng(3)
    x = _f16(rng.standard_normal((5, 256)))
    w = _f16(rng.uniform(0.5, 2.0, 256))
    c, s = oracle.rmsnorm_quantize_rows(x, w, 1e-6)
    cn, sn = oracle.rmsnorm_quantize_rows(x, -w, 1e-6)
    assert np.array_equal(cn, -c) and np.array_equal(sn, s)


def test_zero_rows_give_zero_codes():
    x = np.zeros((3, 64), np.float16)
    for eps in (0.0, 1e-6):
        codes, scale = oracle.rmsnorm_quantize_rows(x, np.ones(64, np.float16), eps)
        assert not codes.any() and not scale.any()


def test_unit_gain_gives_unit_mean_square():
    rng = np.random.default_rng(4)
    x = _f16(rng.standard_normal((4, 4096)) * 3)
    y = oracle.rmsnorm_rows(x, np.ones(4096, np.float16), 0.0).astype(np.float64)
    assert np.allclose((y ** 2).mean(axis=1), 1.0, rtol=2e-3)

"""Pins for the oracle's 4-bit quantizer and code cosine (CPU only).

The quantizer is the paper's W4A4 activation / weight quantizer (App. A,
App. B.3: symmetric, round-to-nearest, one scale per token or per output
channel, clip ratio 1.0) under the fp32 reading. Every expectation below is
computed independently of the oracle: exact rational arithmetic with
``fractions.Fraction``, float64 numpy, or values worked out by hand.
"""
import os
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle


def _f32_neighbors(s: np.float32):
    return (np.nextafter(s, np.float32(-np.inf)), np.nextafter(s, np.float32(np.inf)))


def _rows(seed, rows, cols, outliers=True):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((rows, cols)).astype(np.float32)
    if outliers:
        x[:, rng.choice(cols, min(4, cols), replace=False)] *= 20
    return x.astype(np.float16)


def test_scale_is_correctly_rounded_absmax_over_7():
    x = _rows(1, 64, 257)
    _, s = oracle.quantize_rows(x)
    for r in range(x.shape[0]):
        a = Fraction(float(np.abs(x[r].astype(np.float64)).max()))
        target = a / 7
        err = abs(Fraction(float(s[r])) - target)
        for nb in _f32_neighbors(s[r]):
            assert err <= abs(Fraction(float(nb)) - target)


def test_codes_are_nearest_integers_in_range():
    x = _rows(2, 32, 300)
    c, s = oracle.quantize_rows(x)
    assert c.min() >= -7 and c.max() <= 7
    half = Fraction(1, 2) + Fraction(1, 2 ** 20)  # rounding of the fp32 quotient allowed
    for r in range(x.shape[0]):
        sr = Fraction(float(s[r]))
        for k in range(0, x.shape[1], 7):
            q = Fraction(float(x[r, k])) / sr
            assert abs(q - int(c[r, k])) <= half


def test_absmax_element_maps_to_pm7():
    x = _rows(3, 40, 128)
    c, _ = oracle.quantize_rows(x)
    am = np.abs(x.astype(np.float32)).argmax(axis=1)
    top = c[np.arange(x.shape[0]), am]
    sign = np.sign(x[np.arange(x.shape[0]), am].astype(np.float32))
    assert np.array_equal(top, (7 * sign).astype(np.int8))


def test_zero_row_gives_zero_scale_and_codes():
    x = np.zeros((3, 64), np.float16)
    x[1, 5] = 1.0
    c, s = oracle.quantize_rows(x)
    assert s[0] == 0 and s[2] == 0 and not c[0].any() and not c[2].any()
    assert c[1, 5] == 7 and s[1] > 0


def test_requantizing_the_dequantized_row_keeps_the_codes():
    x = _rows(4, 16, 512)
    c, s = oracle.quantize_rows(x)
    deq = c.astype(np.float64) * s[:, None].astype(np.float64)
    c2, s2 = oracle.quantize_rows(deq.astype(np.float32))
    assert np.array_equal(c, c2)
    np.testing.assert_allclose(s2, s, rtol=2 ** -22)


def test_worked_examples(golden_dir):
    path = os.path.join(golden_dir, "quant_worked_examples.txt")
    n = 0
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        xs, sh, cs = (p.strip() for p in line.split("|"))
        x = np.array([float(v) for v in xs.split()], np.float16)
        want_s = struct.unpack(">f", bytes.fromhex(sh))[0]
        want_c = np.array([int(v) for v in cs.split()], np.int8)
        c, s = oracle.quantize_rows(x[None])
        assert np.float32(s[0]).tobytes() == np.float32(want_s).tobytes(), line
        assert np.array_equal(c[0], want_c), line
        n += 1
    assert n >= 7


def test_pack_unpack_roundtrip():
    rng = np.random.default_rng(5)
    c = rng.integers(-8, 8, size=(7, 64)).astype(np.int8)
    p = oracle.pack_codes(c)
    assert p.shape == (7, 32) and p.dtype == np.uint8
    assert np.array_equal(oracle.unpack_codes(p), c)
    # even index in the low nibble, two's complement
    assert oracle.pack_codes(np.array([[-1, 2]], np.int8))[0, 0] == 0x2F


def test_cosine_matches_float64_of_dequantized_vectors():
    x = _rows(6, 50, 1024)
    c, s = oracle.quantize_rows(x)
    deq = c.astype(np.float64) * s[:, None].astype(np.float64)
    for i in range(0, 50, 3):
        for j in range(1, 50, 5):
            ref = deq[i] @ deq[j] / (np.linalg.norm(deq[i]) * np.linalg.norm(deq[j]))
            got = oracle.cosine(c[i], c[j])
            assert abs(float(got) - ref) <= 2e-6, (i, j, got, ref)


def test_cosine_special_cases():
    d = 64
    a = np.zeros(d, np.int8); a[3] = 5
    b = np.zeros(d, np.int8); b[7] = -2
    assert oracle.cosine(a, b) == 0.0            # orthogonal
    v = np.random.default_rng(7).integers(-7, 8, size=d).astype(np.int8)
    assert abs(float(oracle.cosine(v, v)) - 1.0) <= 2 ** -23
    assert abs(float(oracle.cosine(v, -v)) + 1.0) <= 2 ** -23
    assert oracle.cosine(v, np.zeros(d, np.int8)) == 0.0   # zero vector


@pytest.mark.parametrize("planted", ["drop_round", "reciprocal", "exact_rational"])
def test_worked_examples_reject_a_planted_quantizer_mistake(planted, golden_dir):
    """A wrong quantizer (truncation, multiply by 7/a, or rounding the exact
    rational quotient) disagrees with at least one worked example."""
    rows = []
    for line in open(os.path.join(golden_dir, "quant_worked_examples.txt")):
        line = line.strip()
        if line and not line.startswith("#"):
            xs, _, cs = (p.strip() for p in line.split("|"))
            rows.append((np.array([float(v) for v in xs.split()], np.float32),
                         np.array([int(v) for v in cs.split()], np.int8)))
    differs = False
    for x, want in rows:
        a = np.abs(x).max()
        if a == 0:
            continue
        if planted == "drop_round":
            bad = np.trunc(x / (a / np.float32(7)))
        elif planted == "reciprocal":
            bad = np.rint(x * (np.float32(7) / a))
        else:
            s = Fraction(float(a / np.float32(7)))
            bad = np.array([float(round(Fraction(float(v)) / s)) for v in x])
        differs |= not np.array_equal(bad.astype(np.int8), want)
    assert differs

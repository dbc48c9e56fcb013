"""Comparison helpers shared by the parity tests (test code only).

The tolerance is the one stated for dequantized fp16 outputs: within 1e-3
relative error of the oracle's fp32 dequant, with a 2e-3 absolute floor.
Codes and scales compare bit for bit.
"""
import numpy as np
import torch

import oracle

RTOL, ATOL = 1e-3, 2e-3


def assert_close(y16, ref):
    y = y16.astype(np.float32)
    err = np.abs(y - ref)
    bad = err > np.maximum(ATOL, RTOL * np.abs(ref))
    assert not bad.any(), f"{int(bad.sum())} of {bad.size} outputs outside tolerance (max |err| {err.max()})"


def assert_codes_equal(packed, scales, codes_ref, scales_ref):
    assert np.array_equal(oracle.unpack_codes(packed), codes_ref)
    assert np.array_equal(np.ascontiguousarray(scales).view(np.uint32), scales_ref.view(np.uint32))


def codes_from_expanded(u):
    """Codes in natural order from expanded bytes u = code + 8, stored per 8
    codes as the four even-index codes, then the four odd-index codes."""
    u = np.asarray(u, dtype=np.int16).reshape(u.shape[0], -1, 8) - 8
    out = np.empty_like(u)
    out[:, :, 0::2] = u[:, :, :4]
    out[:, :, 1::2] = u[:, :, 4:]
    return out.reshape(u.shape[0], -1).astype(np.int8)


def assert_expanded_codes_equal(u, sums, scales, codes_ref, scales_ref):
    codes = codes_from_expanded(u)
    assert np.array_equal(codes, codes_ref)
    assert np.array_equal(np.asarray(sums), (codes.astype(np.int64) + 8).sum(axis=1))
    assert np.array_equal(np.ascontiguousarray(scales).view(np.uint32), scales_ref.view(np.uint32))


def sample_rows(M, n, seed):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, M - 1], rng.choice(M, size=min(M, n), replace=False)]))


def take(t, rows):
    return t[torch.from_numpy(rows).to(t.device)].cpu().numpy()

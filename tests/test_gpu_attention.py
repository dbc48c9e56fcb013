"""GPU parity of the causal FP16-KV attention on the pruned sequence against
the oracle (fp64). Bound from the kernel's arithmetic: the softmax weights are
rounded to fp16 before the product with V (relative error <= 2^-11 each) and
the output is rounded to fp16, so |o - o*| <= 2^-11 (max|v| + |o*|) plus fp32
terms; the test allows 5.2e-4 (max|v| + |o*|) + 1e-5, max|v| over the
sample's positions of the head."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

DH = 128


def _inputs(B, m, H, Hkv, seed, qscale=1.0):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal((B * m, H * DH)) * qscale).astype(np.float16)
    k = rng.standard_normal((B * m, Hkv * DH)).astype(np.float16)
    v = rng.standard_normal((B * m, Hkv * DH)).astype(np.float16)
    return q, k, v


def _check(got, want, v, B, m, H, Hkv):
    vv = np.abs(v.astype(np.float64)).reshape(B, m, Hkv, DH).max(axis=(1, 3))       # [B, Hkv]
    vmax = np.repeat(vv, H // Hkv, axis=1)                                           # [B, H]
    bound = 5.2e-4 * (np.repeat(vmax[:, None, :, None], m, axis=1) + np.abs(want).reshape(B, m, H, DH)) + 1e-5
    err = np.abs(got.astype(np.float64).reshape(B, m, H, DH) - want.reshape(B, m, H, DH))
    bad = np.argwhere(err > bound)
    assert bad.size == 0, f"{len(bad)} outputs off, first {bad[:3].tolist()}, max err {err.max():.3g}"


def _run(p4q, dev, q, k, v, B, m, H, Hkv, ldo=None):
    Q, K, V = (torch.from_numpy(a).to(dev) for a in (q, k, v))
    ldo = ldo or H * DH
    O = torch.full((B * m, ldo), 7.0, dtype=torch.float16, device=dev)
    p4q.p4q_causal_attention(Q, K, V, O, B, m, H, Hkv)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    out = O.cpu().numpy()
    assert np.all(out[:, H * DH:] == 7.0), "columns past the heads were written"
    return out[:, :H * DH]


@pytest.mark.parametrize("B,m,H,Hkv", [(1, 1, 1, 1), (2, 77, 2, 2), (1, 128, 4, 4), (3, 200, 4, 2),
                                       (2, 384, 3, 3), (5, 129, 2, 1), (2, 320, 2, 2), (1, 257, 2, 2),
                                       (2, 700, 2, 1), (1, 1030, 1, 1)])
def test_attention_matches_oracle(p4q, dev, B, m, H, Hkv):
    q, k, v = _inputs(B, m, H, Hkv, seed=B * 1000 + m)
    got = _run(p4q, dev, q, k, v, B, m, H, Hkv, ldo=H * DH + 64)
    want = oracle.causal_attention(q, k, v, B, m, H, Hkv, DH)
    _check(got, want, v, B, m, H, Hkv)


def test_attention_peaked_rows(p4q, dev):
    """Large logits (one key dominates most rows) and tiny ones (near-uniform
    rows), over one key chunk and over three (the running maximum moves)."""
    for (B, m, H), scale in [((2, 150, 2), 6.0), ((2, 150, 2), 0.01), ((1, 600, 2), 6.0), ((1, 600, 2), 0.01)]:
        q, k, v = _inputs(B, m, H, H, seed=7, qscale=scale)
        got = _run(p4q, dev, q, k, v, B, m, H, H)
        _check(got, oracle.causal_attention(q, k, v, B, m, H, H, DH), v, B, m, H, H)


def test_attention_on_fused_projection_blocks(p4q, dev):
    """q, k, v as column blocks of one fused q|k|v output (row pitch 3 H dh)."""
    B, m, H = 2, 256, 4
    rng = np.random.default_rng(11)
    Y = rng.standard_normal((B * m, 3 * H * DH)).astype(np.float16)
    Yd = torch.from_numpy(Y).to(dev)
    Q, K, V = Yd[:, :H * DH], Yd[:, H * DH:2 * H * DH], Yd[:, 2 * H * DH:]
    O = torch.empty((B * m, H * DH), dtype=torch.float16, device=dev)
    p4q.p4q_causal_attention(Q, K, V, O, B, m, H, H)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    q, k, v = (np.ascontiguousarray(Y[:, i * H * DH:(i + 1) * H * DH]) for i in range(3))
    _check(O.cpu().numpy(), oracle.causal_attention(q, k, v, B, m, H, H, DH), v, B, m, H, H)


@pytest.mark.parametrize("B,m,H", [(8, 256, 32), (16, 384, 32), (8, 704, 40)])
def test_attention_fullsize_sampled(p4q, dev, B, m, H):
    """The LLaVA-1.5-7B (8 x 256) and LLaVA-NeXT-7B (16 x 384) pruned sequences
    with 32 heads, and LLaVA-NeXT-13B's (640 + 64 positions, 40 heads; 8 of its
    32 samples), heads of 128: every output row of sampled (sample, head) pairs."""
    q, k, v = _inputs(B, m, H, H, seed=m)
    got = _run(p4q, dev, q, k, v, B, m, H, H)
    rng = np.random.default_rng(0)
    for b, h in zip(rng.integers(0, B, 4), rng.integers(0, H, 4)):
        rows = slice(b * m, (b + 1) * m)
        cols = slice(h * DH, (h + 1) * DH)
        want = oracle.causal_attention(q[rows, cols], k[rows, cols], v[rows, cols], 1, m, 1, 1, DH)
        _check(got[rows, cols], want, v[rows, cols], 1, m, 1, 1)


def test_attention_many_units_per_cta(p4q, dev):
    """Enough (sample, head) pairs that every persistent CTA works through
    several units of mixed length (three query blocks per sample, the last
    one ragged) and the last group of pairs is partly empty: the O buffers
    and their read-out barriers cycle many times."""
    B, m, H, Hkv = 8, 300, 40, 8  # 960 units on 150 CTAs; 320 pairs in groups of 50
    q, k, v = _inputs(B, m, H, Hkv, seed=31)
    got = _run(p4q, dev, q, k, v, B, m, H, Hkv)
    _check(got, oracle.causal_attention(q, k, v, B, m, H, Hkv, DH), v, B, m, H, Hkv)


def test_attention_longest_sample(p4q, dev):
    """The documented maximum, m = 8192 positions (64 query blocks, up to 64
    key chunks per block): the row sums and P V accumulate over 8192 keys."""
    B, m, H, Hkv = 1, 8192, 1, 1
    q, k, v = _inputs(B, m, H, Hkv, seed=41)
    got = _run(p4q, dev, q, k, v, B, m, H, Hkv)
    _check(got, oracle.causal_attention(q, k, v, B, m, H, Hkv, DH), v, B, m, H, Hkv)

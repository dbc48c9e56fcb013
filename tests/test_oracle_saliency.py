"""Pins of the oracle's CLS-to-patch saliency (Sec. 3.2, Visual Saliency):
closed forms and invariants of the head-averaged softmax attention of each
crop's [CLS] query over its CLS key and patch keys, independent of the
oracle's own loops."""
import math

import numpy as np

import oracle


def _inputs(B, C, n, H, dh, seed):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((B, C, H, dh)).astype(np.float16)
    kc = rng.standard_normal((B, C, H, dh)).astype(np.float16)
    k = rng.standard_normal((B, C * n, H, dh)).astype(np.float16)
    return q, kc, k


def test_two_tokens_one_head_is_a_sigmoid():
    # CLS key and one patch key, integer vectors: logits by hand
    q = np.array([[[[1, 2, 0, -1]]]], np.float16)        # [1, 1, 1, 4]
    kc = np.array([[[[0, 1, 1, 0]]]], np.float16)        # q . kc = 2
    k = np.array([[[[2, 1, 0, 1]]]], np.float16)         # q . k = 3
    A = oracle.cls_saliency(q, kc, k)
    # softmax over {2/2, 3/2}: the patch weight is 1 / (1 + exp(1 - 1.5))
    assert A.shape == (1, 1)
    assert abs(A[0, 0] - 1.0 / (1.0 + math.exp(-0.5))) < 1e-15


def test_heads_are_averaged():
    q = np.array([[[[1, 0], [0, 1]]]], np.float16)       # two heads, dh = 2
    kc = np.zeros((1, 1, 2, 2), np.float16)               # CLS logit 0 in both heads
    k = np.array([[[[2, 0], [0, -2]]]], np.float16)       # head 0 logit 2/sqrt2, head 1 logit -2/sqrt2
    A = oracle.cls_saliency(q, kc, k)
    s = math.sqrt(2.0)
    want = 0.5 * (1.0 / (1.0 + math.exp(-s)) + 1.0 / (1.0 + math.exp(s)))
    assert abs(A[0, 0] - want) < 1e-15
    assert abs(A[0, 0] - 0.5) < 1e-15  # the two heads are mirror images


def test_patch_weights_sum_to_one_without_the_cls_key():
    q, kc, k = _inputs(2, 3, 40, 4, 16, seed=1)
    kc = (-64.0 * q.astype(np.float32)).astype(np.float16)  # CLS logit far below every patch logit
    A = oracle.cls_saliency(q, kc, k)
    sums = A.reshape(2, 3, 40).sum(-1)
    assert np.allclose(sums, 1.0, atol=1e-12)


def test_identical_keys_give_uniform_weights():
    B, C, n, H, dh = 1, 2, 31, 3, 8
    q, _, _ = _inputs(B, C, n, H, dh, seed=2)
    key = np.random.default_rng(3).standard_normal((H, dh)).astype(np.float16)
    kc = np.broadcast_to(key, (B, C, H, dh)).copy()
    k = np.broadcast_to(key, (B, C * n, H, dh)).copy()
    A = oracle.cls_saliency(q, kc, k)
    assert np.allclose(A, 1.0 / (n + 1), rtol=0, atol=1e-15)


def test_permuting_patches_permutes_the_weights():
    q, kc, k = _inputs(1, 1, 50, 4, 16, seed=4)
    perm = np.random.default_rng(5).permutation(50)
    A = oracle.cls_saliency(q, kc, k)
    Ap = oracle.cls_saliency(q, kc, k[:, perm])
    assert np.allclose(Ap[0], A[0, perm], rtol=1e-13, atol=0)


def test_crops_are_independent():
    q, kc, k = _inputs(1, 3, 20, 2, 8, seed=6)
    A = oracle.cls_saliency(q, kc, k)
    k2 = k.copy()
    k2[:, 20:40] = np.random.default_rng(7).standard_normal(k2[:, 20:40].shape).astype(np.float16)
    A2 = oracle.cls_saliency(q, kc, k2)
    assert np.array_equal(A[:, :20], A2[:, :20]) and np.array_equal(A[:, 40:], A2[:, 40:])
    assert not np.array_equal(A[:, 20:40], A2[:, 20:40])


def test_softmax_shift_invariance():
    # adding the same vector component along q to every key (CLS included)
    # shifts every logit of a head by the same amount: the weights do not move
    q, kc, k = _inputs(1, 1, 30, 1, 8, seed=8)
    qq = q.astype(np.float64)[0, 0, 0]
    shift = (4.0 * qq / np.dot(qq, qq)).astype(np.float16)  # fp16 vector; its dot with q is ~4
    A = oracle.cls_saliency(q, kc, k)
    kc2 = (kc.astype(np.float32) + shift.astype(np.float32)).astype(np.float16)
    k2 = (k.astype(np.float32) + shift.astype(np.float32)).astype(np.float16)
    # fp16 rounding of the shifted keys perturbs the logits slightly: compare loosely
    A2 = oracle.cls_saliency(q, kc2, k2)
    assert np.allclose(A2, A, rtol=2e-2, atol=1e-4)

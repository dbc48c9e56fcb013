"""GPU parity of the CLS-to-patch saliency kernel (Sec. 3.2, Visual Saliency)
against the fp64 oracle, and of the selector fed with it."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

# fp32 logits (dh fp16 products accumulated in fp32), expf, one division per
# head and an fp32 head average: relative error a few ulp of fp32 on weights
# of order 1 / (n + 1).
RTOL, ATOL = 2e-5, 1e-9


def _t(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def _check(p4q, dev, q, kc, k):
    A = p4q.cls_saliency(_t(q, dev), _t(kc, dev), _t(k, dev))
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    got = A.cpu().numpy()
    ref = oracle.cls_saliency(q, kc, k)
    err = np.abs(got - ref)
    assert np.all(err <= ATOL + RTOL * np.abs(ref)), f"max rel err {np.max(err / np.maximum(ref, 1e-30))}"
    return got


@pytest.mark.parametrize("B,N,crop", [(2, 576, 576), (2, 2880, 576), (1, 576, 576)])
def test_saliency_llava_crops(p4q, dev, B, N, crop):
    """One 576-token crop (LLaVA-1.5) and five (LLaVA-NeXT), 16 heads x 64."""
    v = wl.vision_attention(B, N, seed=B + N)
    got = _check(p4q, dev, v.q_cls, v.k_cls, v.k)
    C = N // crop
    assert np.all(got.reshape(B, C, crop).sum(-1) < 1.0)  # the CLS key keeps part of each row


@pytest.mark.parametrize("H,dh,n,C", [(3, 32, 100, 1), (5, 80, 64, 2), (16, 128, 37, 3), (32, 64, 50, 1),
                                      (1, 64, 1, 4)])
def test_saliency_shapes(p4q, dev, H, dh, n, C):
    """Ragged token counts (not multiples of 32), every head dimension, more
    heads than warps, one-token crops."""
    rng = np.random.default_rng(H * 100 + dh + n)
    q = (rng.standard_normal((2, C, H, dh)) * 2).astype(np.float16)
    kc = rng.standard_normal((2, C, H, dh)).astype(np.float16)
    k = rng.standard_normal((2, C * n, H, dh)).astype(np.float16)
    _check(p4q, dev, q, kc, k)


def test_saliency_feeds_the_selector(p4q, dev):
    """A_cls from the kernel drives stage 2: the selector's picks equal the
    oracle's on the same A_cls."""
    w = wl.Workload("t", B=2, N=576, d=512, K=64, T=0, J=3, seed=11, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    v = wl.vision_attention(w.B, w.N, seed=12)
    A = p4q.cls_saliency(_t(v.q_cls, dev), _t(v.k_cls, dev), _t(v.k, dev))
    idx = p4q.select(_t(x.V, dev), _t(x.Q, dev), A, w.K)
    torch.cuda.synchronize()
    ref = oracle.select_batch(x.V, w.K, x.Q, A.cpu().numpy())
    assert np.array_equal(idx.cpu().numpy(), ref)

"""Parity over the GEMM + quantizer sweep and the selector sweep.

GEMM + quantizer: M in {16, 64, 256, 1024, 4096, 16384, 65536} rows x
(K_in, N_out) in {(4096, 4096), (4096, 11008), (11008, 4096), (5120, 13824)}.
The activations of every M are the first M rows of one 65536-row draw per
K_in (fp16 N(0, 1) with the outlier channels); weights N(0, 0.02) with
per-output-channel INT4 (App. B.3). Every weight's codes and scales are
bit-exact; for each shape the activation codes and scales of the checked rows
(every row up to M = 64, else first, last and random rows) are bit-exact and
their fp16 outputs are within tolerance of the oracle's fp32 dequant.

Selector: one grid point per token count of the sweep (576 to 2880 tokens,
1 to 64 images, budgets 5% to 50% of N; Sec. 3.2, Eq. 4); sampled images
against the oracle, every image for the index-set properties.
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl
from parity import assert_close, assert_codes_equal, sample_rows, take

pytestmark = pytest.mark.gpu


@functools.lru_cache(maxsize=1)
def activations(k_in):
    return wl.activations(max(wl.SWEEP_M), k_in, seed=wl.SWEEP_SEED)


@pytest.mark.parametrize("kn", range(len(wl.SWEEP_KN)), ids=[f"{k}x{n}" for k, n in wl.SWEEP_KN])
def test_gemm_quant_sweep(p4q, dev, kn):
    k_in, n_out = wl.SWEEP_KN[kn]
    W = wl.weight(k_in, n_out, wl.weight_seed(wl.SWEEP_SEED, kn))
    Wq, sw = p4q.quant_weight(torch.from_numpy(W).to(dev))
    cw, sw_ref = oracle.quantize_rows(W)
    assert_codes_equal(Wq.cpu().numpy(), sw.cpu().numpy(), cw, sw_ref)
    Xh = activations(k_in)
    Xd = torch.from_numpy(Xh).to(dev)
    for M in wl.SWEEP_M:
        Xq, s = p4q.quant_act(Xd[:M])
        Y = p4q.w4a4_linear(Xq, s, Wq, sw)
        torch.cuda.synchronize()
        assert p4q.p4q_device_status() == 0
        rows = np.arange(M) if M <= 64 else sample_rows(M, 24, M + kn)
        c, sc = oracle.quantize_rows(Xh[rows])
        assert_codes_equal(take(Xq, rows), take(s, rows), c, sc)
        assert_close(take(Y, rows), oracle.linear(c, sc, cw, sw_ref))
        del Xq, s, Y
    del Xd
    torch.cuda.empty_cache()


SELECTOR_POINTS = [  # (N, B, budget %, images checked against the oracle)
    (576, 64, 5.0, [0, 63]),
    (1152, 16, 10.0, [0, 15]),
    (1728, 4, 25.0, [0, 3]),
    (2304, 1, 11.1, [0]),
    (2880, 4, 50.0, [3]),
]


@pytest.mark.parametrize("N,B,pct,images", SELECTOR_POINTS,
                         ids=[f"n{n}-b{b}-{p:g}pct" for n, b, p, _ in SELECTOR_POINTS])
def test_selector_sweep(p4q, dev, N, B, pct, images):
    w = wl.sweep_selector_workload(N, B, pct)
    x = wl.selector_inputs(w)
    idx = p4q.select(torch.from_numpy(x.V).to(dev), torch.from_numpy(x.Q).to(dev), torch.from_numpy(x.A).to(dev),
                     w.K)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    idx = idx.cpu().numpy()
    assert idx.shape == (B, w.K)
    assert (idx >= 0).all() and (idx < N).all() and (np.diff(idx, axis=1) > 0).all()
    ref = oracle.select_batch(x.V[images], w.K, x.Q[images], x.A[images])
    assert np.array_equal(idx[images], ref)
    torch.cuda.empty_cache()

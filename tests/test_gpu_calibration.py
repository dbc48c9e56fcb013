"""GPU parity of the pruning-aware calibration data path against the oracle:
Eq. 5's block objective (Sec. 3.3; per-sample ||Yq - Yf||_F^2 / (m_n d) and
the batch mean, within 1e-5 relative of the fp64 oracle on the same fp16
outputs: fp32 squares summed over a few hundred values per thread, fp64
beyond), Eq. 9's Top-K replacement ratio (App. A; intersection counts and
ratio bits exact), and the whole path on a small batch: selector -> FP16
pruned sequence -> W4A4 block and full-precision block -> objective."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _mse(p4q, dev, Yq, Yf, off):
    B = len(off) - 1
    e = torch.empty((B,), dtype=torch.float32, device=dev)
    L = torch.empty((1,), dtype=torch.float32, device=dev)
    ws = torch.empty((p4q.p4q_block_mse_workspace_bytes(B),), dtype=torch.uint8, device=dev)
    p4q.p4q_block_mse(Yq, Yf, off, e, L, ws)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    return e.cpu().numpy(), float(L.cpu()[0])


def _close(got, want, rtol=1e-5):
    want = np.asarray(want, np.float64)
    assert np.all(np.abs(np.asarray(got, np.float64) - want) <= rtol * np.abs(want) + 1e-30), (got, want)


@pytest.mark.parametrize("lens,d", [([256] * 8, 4096), ([1, 77, 300, 5], 64), ([3] * 1024, 16),
                                    ([2880 + 64], 128), ([384] * 16, 4096)])
def test_block_mse_matches_oracle(p4q, dev, lens, d):
    rng = np.random.default_rng(len(lens) * 10 + d)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    Yq = rng.standard_normal((off[-1], d)).astype(np.float16)
    Yf = (Yq.astype(np.float32) + 0.05 * rng.standard_normal(Yq.shape)).astype(np.float16)
    e, L = _mse(p4q, dev, torch.from_numpy(Yq).to(dev), torch.from_numpy(Yf).to(dev), off.tolist())
    e_ref, L_ref = oracle.block_mse(Yq, Yf, off)
    _close(e, e_ref)
    _close([L], [L_ref])


def test_block_mse_identical_outputs_and_row_pitch(p4q, dev):
    rng = np.random.default_rng(3)
    W = rng.standard_normal((500, 3 * 256)).astype(np.float16)
    Wd = torch.from_numpy(W).to(dev)
    off = [0, 100, 250, 500]
    e, L = _mse(p4q, dev, Wd[:, :256], Wd[:, :256], off)
    assert not e.any() and L == 0.0
    e, L = _mse(p4q, dev, Wd[:, 256:512], Wd[:, 512:], off)  # column blocks, row pitch 768
    e_ref, L_ref = oracle.block_mse(W[:, 256:512], W[:, 512:], off)
    _close(e, e_ref)
    _close([L], [L_ref])


@pytest.mark.parametrize("B,N,K", [(1, 1, 1), (4, 77, 10), (8, 576, 64), (3, 2880, 320), (2, 4096, 4096),
                                   (5, 300, 150), (64, 576, 57)])
def test_topk_replacement_matches_oracle(p4q, dev, B, N, K):
    rng = np.random.default_rng(B * 7 + N)
    s_ref = rng.standard_normal((B, N)).astype(np.float32)
    s_alt = (s_ref + 0.5 * rng.standard_normal((B, N))).astype(np.float32)
    s_ref[:, ::5] = 0.0                      # ties at zero, with -0 and +0 mixed
    s_alt[:, 1::5] = -0.0
    s_alt[:, 2::5] = 0.0
    s_ref[:, 3::11] = s_ref[:, 3:4]          # ties at a non-zero value
    inter = torch.empty((B,), dtype=torch.int32, device=dev)
    rho = torch.empty((B,), dtype=torch.float32, device=dev)
    p4q.p4q_topk_replacement(torch.from_numpy(s_ref).to(dev), torch.from_numpy(s_alt).to(dev), K, inter, rho)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    i_ref, r_ref = oracle.topk_replacement(s_ref, s_alt, K)
    assert np.array_equal(inter.cpu().numpy(), i_ref)
    assert np.array_equal(rho.cpu().numpy().view(np.uint32), r_ref.view(np.uint32))


def test_calibration_path_end_to_end(p4q, dev):
    """Selector -> H^{FP,keep} (X) -> W4A4 block (p4q) and full-precision block
    (the same weights in fp16, a library matmul) -> Eq. 5 objective, against
    the oracle's chain with a float64 full-precision block."""
    w = wl.Workload("calib", B=3, N=320, d=512, K=48, T=16, J=3, seed=11, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    W = wl.weight(w.d, 256, seed=5)
    Vd, Qd, Ad, Td = (torch.from_numpy(a).to(dev) for a in (x.V, x.Q, x.A, x.text))
    idx, X, Xq, s_a = p4q.select_gather_quant(Vd, Qd, Ad, Td, w.K)
    Wd = torch.from_numpy(W).to(dev)
    Wq, s_w = p4q.quant_weight(Wd)
    Yq = p4q.w4a4_linear(Xq, s_a, Wq, s_w)
    H = X.reshape(-1, w.d)
    Yf = (H.float() @ Wd.float().t()).to(torch.float16)
    m = w.K + w.T
    off = [n * m for n in range(w.B + 1)]
    e, L = _mse(p4q, dev, Yq, Yf, off)
    # the kernel on the same outputs
    e_ref, L_ref = oracle.block_mse(Yq.cpu().numpy(), Yf.cpu().numpy(), off)
    _close(e, e_ref)
    _close([L], [L_ref])
    # the oracle's whole chain
    ref_idx = oracle.select_batch(x.V, w.K, x.Q, x.A)
    assert np.array_equal(idx.cpu().numpy(), ref_idx)
    Hr = oracle.gather(x.V, ref_idx, x.text).reshape(-1, w.d)
    ca, sa = oracle.quantize_rows(Hr)
    cw, sw = oracle.quantize_rows(W)
    Yq_ref = oracle.linear(ca, sa, cw, sw)
    Yf_ref = Hr.astype(np.float64) @ W.astype(np.float64).T
    e2, L2 = oracle.block_mse(Yq_ref, Yf_ref.astype(np.float32), off)
    assert abs(L - L2) <= 2e-2 * L2 and np.all(np.abs(e - e2) <= 2e-2 * e2)

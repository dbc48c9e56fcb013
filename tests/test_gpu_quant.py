"""GPU parity of the per-row INT4 quantizer (App. A / App. B.3) against the
oracle: packed codes and fp32 scale bits must be bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _run(p4q, dev, x):
    X = torch.from_numpy(x).to(dev)
    Xq, s = p4q.quant_act(X)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    return Xq.cpu().numpy(), s.cpu().numpy()


def _check(p4q, dev, x):
    q, s = _run(p4q, dev, x)
    c, sr = oracle.quantize_rows(x)
    assert np.array_equal(s.view(np.uint32), sr.view(np.uint32)), "scale bits differ"
    got = oracle.unpack_codes(q)
    bad = np.argwhere(got != c)
    assert bad.size == 0, f"{len(bad)} codes differ, first at {bad[:3].tolist()}"


@pytest.mark.parametrize("M,K", [(1, 16), (7, 128), (33, 4096), (96, 4096), (300, 11008), (17, 13824),
                                 (5, 16384), (257, 5120),
                                 (2100, 5120), (2049, 11008)])  # from 2048 rows: the register-resident kernel
def test_quant_act_matches_oracle(p4q, dev, M, K):
    _check(p4q, dev, wl.activations(M, K, seed=M + K))


def test_quant_heavy_tail_and_zero_rows(p4q, dev):
    x = wl.activations(64, 5120, seed=3, heavy_tail=True)
    x[5] = 0
    x[17, :] = 0
    x[17, 4000] = -0.0
    _check(p4q, dev, x)


def test_quant_worked_example_ties(p4q, dev, golden_dir):
    import os
    rows = []
    for line in open(os.path.join(golden_dir, "quant_worked_examples.txt")):
        line = line.strip()
        if line and not line.startswith("#"):
            xs = [float(v) for v in line.split("|")[0].split()]
            rows.append(xs + [0.0] * (16 - len(xs)))
    _check(p4q, dev, np.array(rows, np.float16))


def test_quant_weight_matches_oracle(p4q, dev):
    W = wl.weight(4096, 136, seed=5)
    Wt = torch.from_numpy(W).to(dev)
    Wq, s = p4q.quant_weight(Wt)
    c, sr = oracle.quantize_rows(W)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), sr.view(np.uint32))
    assert np.array_equal(oracle.unpack_codes(Wq.cpu().numpy()), c)


def test_quant_empty_is_noop(p4q, dev):
    X = torch.empty((0, 128), dtype=torch.float16, device=dev)
    Xq = torch.empty((0, 64), dtype=torch.uint8, device=dev)
    s = torch.empty((0,), dtype=torch.float32, device=dev)
    p4q.p4q_quant_act(X, Xq, s)


def test_quant_rows_full_of_exact_ties(p4q, dev):
    """Rows whose quotients x / s land on exact .5 boundaries (s = 1 or 2^k),
    plus rows near them: the rounding decisions must match the oracle's."""
    rng = np.random.default_rng(21)
    x = (rng.integers(-28, 29, size=(64, 512)) * 0.25).astype(np.float32)
    x[:, 0] = 7.0                      # absmax 7 -> s = 1 exactly
    x[32:] *= np.float32(2.0 ** -3)    # s = 2^-3
    x[48:, 1:] = np.nextafter(x[48:, 1:], np.float32(np.inf))  # just off the boundaries
    _check(p4q, dev, x.astype(np.float16))


def test_quant_act_on_a_column_block_matches_dense(p4q, dev):
    """p4q_quant_act_ld on the middle column block of a wider matrix equals
    p4q_quant_act on a dense copy of that block (and the oracle)."""
    X = torch.from_numpy(wl.activations(300, 3 * 1024, seed=21)).to(dev)
    block = X[:, 1024:2048]
    Xq = torch.empty((300, 512), dtype=torch.uint8, device=dev)
    s = torch.empty((300,), dtype=torch.float32, device=dev)
    p4q.p4q_quant_act_ld(block, Xq, s)
    ref_q, ref_s = p4q.quant_act(block.contiguous())
    torch.cuda.synchronize()
    assert torch.equal(Xq, ref_q) and torch.equal(s.view(torch.int32), ref_s.view(torch.int32))
    c, sc = oracle.quantize_rows(block.cpu().numpy())
    assert np.array_equal(oracle.unpack_codes(Xq.cpu().numpy()), c)


def test_quant_act_expanded_matches_quant_then_expand(p4q, dev):
    """The quantizer's expanded output equals p4q_expand_codes of its packed
    codes (bytes and row sums), for one-warp and multi-warp row lengths."""
    for M, K, seed in [(300, 1024, 31), (77, 11008, 32), (129, 5120, 33), (2048, 5120, 34), (2053, 13824, 35)]:
        X = torch.from_numpy(wl.activations(M, K, seed=seed)).to(dev)
        X[3].zero_()
        Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        Xu = torch.empty((M, K), dtype=torch.uint8, device=dev)
        su = torch.empty((M,), dtype=torch.int32, device=dev)
        p4q.p4q_quant_act_expanded(X, Xq, s, Xu, su)
        ref_q, ref_s = p4q.quant_act(X)
        ref_u, ref_su = p4q.expand_codes(ref_q)
        torch.cuda.synchronize()
        assert torch.equal(Xq, ref_q) and torch.equal(s.view(torch.int32), ref_s.view(torch.int32))
        assert torch.equal(Xu, ref_u) and torch.equal(su, ref_su)

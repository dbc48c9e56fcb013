"""Parity at the full sizes of the LLaVA-shaped workloads, in the launch
configuration bench.py times.

Each test builds bench.Step for the workload (p4q_select_gather_quant with a
caller workspace, the W4A4 linears on the pruned sequence with q|k|v and
gate|up each run as one GEMM over their concatenated output channels, the
re-quantizations of column blocks that feed o and down), runs it once as
plain calls, captures
it as CUDA graphs, clears every output and replays the graphs once: the
outputs checked are those of the replay.

Checked against the oracle:
- kept index sets: every image of the 1- and 8-image batches; the first and
  last image of the 2880-token batches (the oracle needs seconds per image
  there); every image for what holds at any size (K distinct ascending
  indices in range);
- gathered fp16 rows: every row, bit-exact against V[idx] and the text;
- INT4 codes and scales of the pruned sequence, of every weight and of the
  re-quantized o / down inputs: bit-exact (every row; sampled rows for
  re-quantized inputs of more than 64 M elements);
- fp16 outputs of every linear of the last layer: sampled rows (first, last
  and random) within 1e-3 relative / 2e-3 absolute of the oracle's fp32
  dequant (App. B.3).
"""
import dataclasses
import gc

import numpy as np
import pytest
import torch

import bench
import oracle
from paper_2609_34867_gb300 import workloads as wl
from parity import assert_close, assert_codes_equal, assert_expanded_codes_equal, sample_rows, take

pytestmark = pytest.mark.gpu

@pytest.fixture
def run_step(p4q, dev):
    made = []

    def run(w):
        step = bench.Step(w, dev, seed=w.seed)
        step.body()
        torch.cuda.synchronize()
        step.capture()
        for t in [step.X, step.Xq, step.s_a, step.Xu, step.sXu] + list(step.Y.values()) + list(step.Xq_re.values()) + \
                list(step.s_re.values()) + list(step.Xu_re.values()) + list(step.sXu_re.values()):
            t.zero_()
        step.idx.fill_(-1)
        step()
        torch.cuda.synchronize()
        assert p4q.p4q_device_status() == 0
        made.append(step)
        return step

    yield run
    made.clear()
    gc.collect()  # the steps' CUDA graphs go now, not inside a later capture
    torch.cuda.empty_cache()


def check_step(step, w, images, rows):
    x = step.host
    B, K, d = w.B, w.K, w.d
    idx = step.idx.cpu().numpy()
    assert idx.shape == (B, K)
    assert (idx >= 0).all() and (idx < w.N).all()
    assert (np.diff(idx, axis=1) > 0).all()
    ref = oracle.select_batch(x["V"][images], K, x["Q"][images], x["A"][images])
    assert np.array_equal(idx[images], ref)

    gi = step.idx.long()[:, :, None].expand(-1, -1, d)
    assert torch.equal(step.X[:, :K].view(torch.int16), torch.gather(step.V, 1, gi).view(torch.int16))
    assert torch.equal(step.X[:, K:].view(torch.int16), step.text.view(torch.int16))

    ca, sa = oracle.quantize_rows(step.X.reshape(-1, d).cpu().numpy())
    # the step writes the pruned sequence's expanded codes (what its GEMMs read)
    assert_expanded_codes_equal(step.Xu.cpu().numpy(), step.sXu.cpu().numpy(), step.s_a.cpu().numpy(), ca, sa)

    layer = w.layers - 1  # Y holds the last layer's outputs
    for lid, lin in enumerate(w.linears):
        W = wl.weight(lin.k_in, lin.n_out, wl.weight_seed(w.seed + layer, lid))
        cw, sw = oracle.quantize_rows(W)
        Wq, s_w = step.weight(layer, lin.name)
        assert_codes_equal(Wq.cpu().numpy(), s_w.cpu().numpy(), cw, sw)
        if lin.name in step.REQUANT:
            Yin = step.output(step.REQUANT[lin.name])
            every = Yin.numel() <= (64 << 20)
            r = np.arange(w.M) if every else rows
            cq, sq = oracle.quantize_rows(take(Yin, r))
            if step.packed_requant:
                assert_codes_equal(take(step.Xq_re[lin.name], r), take(step.s_re[lin.name], r), cq, sq)
            else:  # the step writes only the expanded codes its GEMM reads
                assert_expanded_codes_equal(take(step.Xu_re[lin.name], r), take(step.sXu_re[lin.name], r),
                                            take(step.s_re[lin.name], r), cq, sq)
            a, s = (cq[rows], sq[rows]) if every else (cq, sq)
        else:
            a, s = ca[rows], sa[rows]
        assert_close(take(step.output(lin.name), rows), oracle.linear(a, s, cw, sw))


def test_one_image_576_to_64(run_step):
    w = wl.LLAVA15_7B_ONE
    check_step(run_step(w), w, images=[0], rows=np.arange(w.M))


def test_llava15_7b_batch_8x576_to_192(run_step):
    w = wl.LLAVA15_7B
    check_step(run_step(w), w, images=list(range(w.B)), rows=sample_rows(w.M, 62, 1))


def spread(B, n=4):
    """n image indices spread across a batch of B, first and last included."""
    return sorted({round(i * (B - 1) / (n - 1)) for i in range(n)})


def test_llavanext_7b_batch_16x2880_to_320(run_step):
    # two of the 32 layers: every layer launches the same kernels on the same
    # shapes, and the second checks that the layer chain reads its own weights
    w = dataclasses.replace(wl.LLAVANEXT_7B, layers=2)
    check_step(run_step(w), w, images=spread(w.B), rows=sample_rows(w.M, 46, 2))


def test_llavanext_13b_batch_32x2880_to_640_heavy_tails(run_step):
    w = wl.LLAVANEXT_13B
    check_step(run_step(w), w, images=spread(w.B), rows=sample_rows(w.M, 30, 3))

"""GPU checks of the single-pass re-quantization of GEMM outputs (App. A:
every linear's input is quantized per token, so the q and up blocks of the
fused q|k|v|gate|up output are re-quantized for o and down): the GEMM's
row-max epilogue gives every row's abs-max per column block, and the
known-max quantizer then writes the same codes, scales, expanded codes and
row sums, bit for bit, as the two-pass quantizer p4q_quant_act_expanded
(itself bit-exact against the oracle in tests/test_gpu_quant.py); codes are
also checked against the oracle directly."""
import numpy as np
import pytest
import torch

import oracle
from parity import assert_codes_equal

pytestmark = pytest.mark.gpu


def _operands(p4q, dev, M, N, K, seed):
    g = torch.Generator(device=dev).manual_seed(seed)
    X = (torch.randn((M, K), generator=g, device=dev) * 2.0).to(torch.float16)
    W = (torch.randn((N, K), generator=g, device=dev) * 0.02).to(torch.float16)
    Xq, s_a = p4q.quant_act(X)
    Wq, s_w = p4q.quant_act(W)
    Xu, sXu = p4q.expand_codes(Xq)
    Wu, sWu = p4q.expand_codes(Wq)
    return Xu, sXu, s_a, Wu, sWu, s_w


def _rowmax_ref(Y, c0, n):
    return (Y[:, c0:c0 + n].contiguous().view(torch.int16).to(torch.int32) & 0x7FFF).amax(dim=1)


@pytest.mark.parametrize("M,N,K,blocks", [(77, 1280, 256, [(0, 256), (768, 512)]),
                                          (2048, 2304, 512, [(0, 512), (1536, 768)]),
                                          (600, 512, 128, [(256, 256)]),
                                          (513, 768, 384, [(32, 96), (224, 544)])])
def test_gemm_rowmax_epilogue(p4q, dev, M, N, K, blocks):
    ops = _operands(p4q, dev, M, N, K, seed=M + N)
    Y0 = torch.empty((M, N), dtype=torch.float16, device=dev)
    p4q.p4q_w4a4_linear_expanded(*ops, Y0)
    Y = torch.full((M, N), float("nan"), dtype=torch.float16, device=dev)
    rowmax = torch.full((len(blocks), M), 12345, dtype=torch.int32, device=dev)  # cleared by the call
    p4q.p4q_w4a4_linear_expanded_rowmax(*ops, Y, blocks, rowmax)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    assert torch.equal(Y.view(torch.int16), Y0.view(torch.int16))  # same GEMM output bit for bit
    for b, (c0, n) in enumerate(blocks):
        assert torch.equal(rowmax[b], _rowmax_ref(Y, c0, n))


def _quant_ref(p4q, Yb):
    M, L = Yb.shape
    Xq = torch.empty((M, L // 2), dtype=torch.uint8, device=Yb.device)
    s = torch.empty((M,), dtype=torch.float32, device=Yb.device)
    Xu = torch.empty((M, L), dtype=torch.uint8, device=Yb.device)
    su = torch.empty((M,), dtype=torch.int32, device=Yb.device)
    p4q.p4q_quant_act_expanded(Yb, Xq, s, Xu, su)
    return Xq, s, Xu, su


@pytest.mark.parametrize("M,ldy,blocks,packed", [(33, 2048, [(0, 512), (768, 1280)], True),
                                                 (2048, 4096 * 3 + 11008 * 2, [(0, 4096), (23296, 11008)], True),
                                                 (300, 1024, [(256, 768)], False),
                                                 (5, 5120, [(0, 5120), (0, 5120)], True),
                                                 (5000, 1536, [(0, 512), (1024, 512)], True),  # one warp per row
                                                 (2048, 6144, [(2048, 4096)], True),           # two warps per row
                                                 (1000, 12032, [(1024, 11008)], False)])       # four, 43 steps
def test_known_max_quantizer_matches_two_pass(p4q, dev, M, ldy, blocks, packed):
    g = torch.Generator(device=dev).manual_seed(M)
    Y = (torch.randn((M, ldy), generator=g, device=dev) * 3.0).to(torch.float16)
    Y[1] = 0.0                                           # a zero row: scale 0, zero codes
    Y[2, ::7] = 60000.0                                  # near the fp16 range
    Y[3] = torch.round(Y[3] * 2.0) / 2.0                 # many exact .5 quotients
    rowmax = torch.stack([_rowmax_ref(Y, c0, n) for c0, n in blocks])
    outs = []
    for c0, n in blocks:
        outs.append((torch.empty((M, n // 2), dtype=torch.uint8, device=dev) if packed else None,
                     torch.empty((M,), dtype=torch.float32, device=dev),
                     torch.empty((M, n), dtype=torch.uint8, device=dev),
                     torch.empty((M,), dtype=torch.int32, device=dev)))
    p4q.p4q_quant_act_expanded_rowmax(Y, blocks, rowmax, [o[0] for o in outs] if packed else None,
                                      [o[1] for o in outs], [o[2] for o in outs], [o[3] for o in outs])
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    for (c0, n), (Xq, s, Xu, su) in zip(blocks, outs):
        rq, rs, ru, rsu = _quant_ref(p4q, Y[:, c0:c0 + n])
        assert torch.equal(s.view(torch.int32), rs.view(torch.int32))
        assert torch.equal(Xu, ru) and torch.equal(su, rsu)
        if packed:
            assert torch.equal(Xq, rq)
    # and the codes of the first block against the oracle
    c0, n = blocks[0]
    r = np.arange(min(M, 64))
    cq, sq = oracle.quantize_rows(Y[r][:, c0:c0 + n].float().cpu().numpy())
    if packed:
        assert_codes_equal(outs[0][0][r].cpu().numpy(), outs[0][1][r].cpu().numpy(), cq, sq)


def test_requant_chain_matches_the_two_pass_chain(p4q, dev):
    """q|k|v|gate|up-shaped GEMM with the row-max epilogue on its q and up
    blocks, then the one-pass quantizer: equal to quantizing the blocks of the
    plain GEMM's output with the two-pass quantizer."""
    M, K, d, ffn = 2048, 512, 512, 1024
    N = 3 * d + 2 * ffn
    blocks = [(0, d), (3 * d + ffn, ffn)]
    ops = _operands(p4q, dev, M, N, K, seed=5)
    Y = torch.empty((M, N), dtype=torch.float16, device=dev)
    rowmax = torch.empty((2, M), dtype=torch.int32, device=dev)
    p4q.p4q_w4a4_linear_expanded_rowmax(*ops, Y, blocks, rowmax)
    outs = [(torch.empty((M, n // 2), dtype=torch.uint8, device=dev), torch.empty((M,), dtype=torch.float32, device=dev),
             torch.empty((M, n), dtype=torch.uint8, device=dev), torch.empty((M,), dtype=torch.int32, device=dev))
            for _, n in blocks]
    p4q.p4q_quant_act_expanded_rowmax(Y, blocks, rowmax, *[[o[i] for o in outs] for i in range(4)])
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    for (c0, n), (Xq, s, Xu, su) in zip(blocks, outs):
        rq, rs, ru, rsu = _quant_ref(p4q, Y[:, c0:c0 + n])
        assert torch.equal(Xq, rq) and torch.equal(s.view(torch.int32), rs.view(torch.int32))
        assert torch.equal(Xu, ru) and torch.equal(su, rsu)

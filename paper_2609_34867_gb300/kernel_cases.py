"""Single-call cases of the hot path, for profiling and microbenchmarks.

  python -m paper_2609_34867_gb300.kernel_cases gemm M N K [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases gemm8 M N K [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases quant M K [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases {requant,requant1} M L LD [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases select WORKLOAD [B] [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases saliency B N [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases swiglu M K LD [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases rmsnorm M K [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases attn B M H [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases mse B M D [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases topk B N K [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases peak {f8,s8,dp4a} ITERS [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases sweep {gemm,quant,select} [--reps R]
  python -m paper_2609_34867_gb300.kernel_cases hostlink MIB [--reps R]

Each case builds seeded synthetic inputs (workloads.py), makes one untimed
warm-up call of the C-ABI entry point on cuda:0, captures the call in a CUDA
graph, then times `reps` replays (default 3), each after an L2 flush (512 MiB
written, then 512 MiB read), and prints the mean CUDA-event time per call with
the throughput it implies. Under ncu, `-s 1 -c 1` with the kernel's name
selects the first replayed launch.

  gemm    p4q_w4a4_linear on random packed codes: M x K activations,
          N x K weights, fp16 output (2 M N K integer ops per call);
  gemm8   p4q_w4a4_linear_expanded on the same operands expanded once by
          p4q_expand_codes before timing (the GEMM kernel alone);
  quant   p4q_quant_act on M x K fp16 activations with the outlier channels
          (bytes: 2 M K in, M K / 2 + 4 M out);
  requant p4q_quant_act_expanded on the last L columns of an M x LD fp16
          matrix (a linear's output block inside a fused GEMM's output), with
          the expanded codes (bytes: 2 M L in, 3 M L / 2 + 8 M out);
  requant1 p4q_quant_act_expanded_rowmax on the same block with its row
          abs-max given (as a GEMM's row-max epilogue records it), expanded
          codes only (bytes: 2 M L in, M L + 8 M out);
  select  p4q_select_gather_quant on one of the LLaVA-shaped workloads (B:
          its first B images instead of all);
  swiglu  p4q_swiglu_quant_expanded on gate / up, the last 2 K columns of an
          M x LD fp16 matrix (bytes: 4 M K in, 3 M K / 2 + 8 M out);
  rmsnorm p4q_rmsnorm_quant_expanded on M x K fp16 rows with a K-value gain
          (bytes: 2 M K + 2 K in, 3 M K / 2 + 8 M out);
  attn    p4q_causal_attention on B samples of M positions, H heads of 128
          (flops: 2 x 2 x 128 x M (M + 1) / 2 per sample and head, the
          causal Q K^T and P V; bytes: q, k, v in, o out, fp16);
  mse     p4q_block_mse on B samples of M rows x D fp16 (bytes: 4 B M D in);
  topk    p4q_topk_replacement on B x N fp32 score pairs (bytes: 8 B N in);
  peak    p4q_peak_probe: the throughput loop of one integer contraction
          pipe (f8: tcgen05 kind::f8f6f4 MMAs on operands in shared memory;
          s8: mma.sync m16n8k32 s8; dp4a), ITERS rounds (ops = 2 per
          multiply-add, as counted by the probe);
  sweep   the GEMM + quantizer sweep (every M x (K, N) of the LLaVA-shaped
          sweep: the W4A4 linear as called, p4q_w4a4_linear_ws with its
          operand expansion, and the GEMM kernel alone on expanded operands;
          p4q_quant_act on every M x K) or the selector sweep (576 .. 2880
          tokens, 1 .. 64 images, budgets 5 .. 50%, inputs drawn on the GPU
          from a seeded generator: N(0,1) with the 8 outlier channels x20, 3
          concepts, softmax CLS saliency), one table row per point;
  saliency p4q_cls_saliency on B images of N tokens (576-token crops, 16
          heads x 64, the CLIP ViT-L vision tower's final layer; bytes: the
          fp16 keys and queries in, 4 B N out);
  hostlink the copies the end-to-end path makes: MIB MiB from pinned host
          memory to the device, back, and both directions at once on two
          streams (the best of the replays; no graph, no kernel of the
          library).
"""
from __future__ import annotations

import argparse
import dataclasses
import sys

import torch

from . import p4q
from . import workloads as wl

FLUSH_BYTES = 512 << 20


def _timed(fn, reps, dev):
    """Mean CUDA-event milliseconds of fn, replayed from a CUDA graph (so that
    no host work sits between the events), L2 flushed before each replay."""
    w = torch.empty((FLUSH_BYTES,), dtype=torch.uint8, device=dev)
    r = torch.ones((FLUSH_BYTES // 4,), dtype=torch.float32, device=dev)
    fn()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fn()
    total = 0.0
    for _ in range(reps):
        w.zero_()
        r.amax()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        graph.replay()
        b.record()
        torch.cuda.synchronize()
        total += a.elapsed_time(b)
    status = p4q.p4q_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the timed calls")
    return total / reps


PEAK_ITERS = {"f8": 60000, "s8": 20000, "dp4a": 40000}  # a few tens of milliseconds per launch


def peak_tops(kind: str, dev, reps: int = 5, iters: int | None = None) -> float:
    """Best rate in TOPS of `reps` timed launches of one throughput probe
    (p4q_peak_probe) on `dev`, after one untimed launch."""
    sink = torch.zeros((8192,), dtype=torch.int32, device=dev)
    it = iters or PEAK_ITERS[kind]
    p4q.p4q_peak_probe(kind, it, sink)
    torch.cuda.synchronize()
    best = 0.0
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        ops = p4q.p4q_peak_probe(kind, it, sink)
        b.record()
        torch.cuda.synchronize()
        best = max(best, ops / (a.elapsed_time(b) * 1e-3) / 1e12)
    status = p4q.p4q_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the peak probe")
    return best


def _sweep(kind: str, reps: int, dev):
    if kind == "gemm":
        print("| M | K | N | linear (ws, expansion included) us | TOPS | GEMM kernel alone us | TOPS |")
        print("|---|---|---|---|---|---|---|")
        g = torch.Generator(device=dev).manual_seed(wl.SWEEP_SEED)
        for K, N in wl.SWEEP_KN:
            Wq = torch.randint(0, 256, (N, K // 2), dtype=torch.uint8, device=dev, generator=g)
            s_w = torch.rand(N, device=dev, generator=g) * 0.01
            Wu, sW = p4q.expand_codes(Wq)
            for M in wl.SWEEP_M:
                Xq = torch.randint(0, 256, (M, K // 2), dtype=torch.uint8, device=dev, generator=g)
                s_a = torch.rand(M, device=dev, generator=g)
                Y = torch.empty((M, N), dtype=torch.float16, device=dev)
                ws = p4q.linear_workspace(M, N, K, dev)
                t_lin = _timed(lambda: p4q.p4q_w4a4_linear_ws(Xq, s_a, Wq, s_w, Y, ws), reps, dev)
                Xu, sX = p4q.expand_codes(Xq)
                if N >= 256 and M >= 16:
                    t_g = _timed(lambda: p4q.p4q_w4a4_linear_expanded(Xu, sX, s_a, Wu, sW, s_w, Y), reps, dev)
                    g8 = f"{t_g * 1e3:.1f} | {2 * M * N * K / t_g / 1e9:.1f}"
                else:
                    g8 = "- | -"
                print(f"| {M} | {K} | {N} | {t_lin * 1e3:.1f} | {2 * M * N * K / t_lin / 1e9:.1f} | {g8} |", flush=True)
                del Xq, Y, ws, Xu, sX
            del Wq, Wu, sW
    elif kind == "quant":
        print("| M | K | us | GB/s |")
        print("|---|---|---|---|")
        for K in sorted({k for k, _ in wl.SWEEP_KN}):
            Xall = torch.from_numpy(wl.activations(max(wl.SWEEP_M), K, seed=wl.SWEEP_SEED)).to(dev)
            for M in wl.SWEEP_M:
                X = Xall[:M]
                Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
                sc = torch.empty((M,), dtype=torch.float32, device=dev)
                t = _timed(lambda: p4q.p4q_quant_act(X, Xq, sc), reps, dev)
                nbytes = 2 * M * K + M * K // 2 + 4 * M
                print(f"| {M} | {K} | {t * 1e3:.1f} | {nbytes / t / 1e6:.1f} |", flush=True)
            del Xall
    else:
        print("| N | B | budget % | K | us / call | us / image |")
        print("|---|---|---|---|---|---|")
        g = torch.Generator(device=dev).manual_seed(wl.SWEEP_SEED)
        d = 4096
        out_ch = torch.from_numpy(wl.outlier_channels(d)).to(dev)
        points = [(N, B, pct) for N in wl.SWEEP_SEL_N for B in wl.SWEEP_SEL_B for pct in (11.1,)]
        points += [(N, 16, pct) for N in (576, 2880) for pct in wl.SWEEP_SEL_PCT if pct != 11.1]
        for N, B, pct in points:
            V = torch.randn((B, N, d), device=dev, generator=g)
            V[:, :, out_ch] *= 20.0
            V = V.to(torch.float16)
            pick = torch.randint(0, N, (B, 3), device=dev, generator=g)
            Q = (V.float().gather(1, pick[:, :, None].expand(B, 3, d)) +
                 0.5 * torch.randn((B, 3, d), device=dev, generator=g)).to(torch.float16)
            A = torch.softmax(2.0 * torch.randn((B, N), device=dev, generator=g), dim=1)
            K = wl.sweep_budget(N, pct)
            ws = p4q.select_workspace(B, N, d, 3, K, dev)
            idx = torch.empty((B, K), dtype=torch.int32, device=dev)
            t = _timed(lambda: p4q.p4q_select(V, Q, A, K, idx, ws), reps, dev)
            print(f"| {N} | {B} | {pct:g} | {K} | {t * 1e3:.1f} | {t * 1e3 / B:.2f} |", flush=True)
            del V, Q, A, ws, idx


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("case", choices=["gemm", "gemm8", "quant", "requant", "requant1", "select", "saliency", "swiglu", "rmsnorm", "attn",
                                     "mse", "topk", "peak", "sweep", "hostlink"])
    ap.add_argument("args", nargs="+")
    ap.add_argument("--reps", type=int, default=3)
    a = ap.parse_args(argv)
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    p4q.lib()
    if a.case in ("gemm", "gemm8"):
        M, N, K = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        Xq = torch.randint(0, 256, (M, K // 2), dtype=torch.uint8, device=dev, generator=g)
        Wq = torch.randint(0, 256, (N, K // 2), dtype=torch.uint8, device=dev, generator=g)
        s_a = torch.rand(M, device=dev, generator=g)
        s_w = torch.rand(N, device=dev, generator=g) * 0.01
        Y = torch.empty((M, N), dtype=torch.float16, device=dev)
        if a.case == "gemm":
            ms = _timed(lambda: p4q.p4q_w4a4_linear(Xq, s_a, Wq, s_w, Y), a.reps, dev)
        else:
            Xu, sX = p4q.expand_codes(Xq)
            Wu, sW = p4q.expand_codes(Wq)
            ms = _timed(lambda: p4q.p4q_w4a4_linear_expanded(Xu, sX, s_a, Wu, sW, s_w, Y), a.reps, dev)
        print(f"{a.case} {M}x{N}x{K}: {ms * 1e3:.1f} us/call, {2 * M * N * K / ms / 1e9:.1f} TOPS")
    elif a.case == "quant":
        M, K = (int(x) for x in a.args)
        X = torch.from_numpy(wl.activations(M, K, seed=wl.SWEEP_SEED)).to(dev)
        Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        ms = _timed(lambda: p4q.p4q_quant_act(X, Xq, s), a.reps, dev)
        nbytes = 2 * M * K + M * K // 2 + 4 * M
        print(f"quant {M}x{K}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "requant":
        M, L, LD = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        Y = (torch.randn((M, LD), generator=g, device=dev) * 4.0).to(torch.float16)
        X = Y[:, LD - L:]
        Xq = torch.empty((M, L // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        Xu = torch.empty((M, L), dtype=torch.uint8, device=dev)
        su = torch.empty((M,), dtype=torch.int32, device=dev)
        ms = _timed(lambda: p4q.p4q_quant_act_expanded(X, Xq, s, Xu, su), a.reps, dev)
        nbytes = 2 * M * L + 3 * M * L // 2 + 8 * M
        print(f"requant {M}x{L} of {LD}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "requant1":
        M, L, LD = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        Y = (torch.randn((M, LD), generator=g, device=dev) * 4.0).to(torch.float16)
        rowmax = (Y[:, LD - L:].contiguous().view(torch.int16).to(torch.int32) & 0x7FFF).amax(dim=1)[None]
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        Xu = torch.empty((M, L), dtype=torch.uint8, device=dev)
        su = torch.empty((M,), dtype=torch.int32, device=dev)
        ms = _timed(lambda: p4q.p4q_quant_act_expanded_rowmax(Y, [(LD - L, L)], rowmax, None, [s], [Xu], [su]),
                    a.reps, dev)
        nbytes = 2 * M * L + M * L + 8 * M
        print(f"requant1 {M}x{L} of {LD}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "swiglu":
        M, K, LD = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        Y = (torch.randn((M, LD), generator=g, device=dev) * 3.0).to(torch.float16)
        G, U = Y[:, LD - 2 * K:LD - K], Y[:, LD - K:]
        Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        Xu = torch.empty((M, K), dtype=torch.uint8, device=dev)
        su = torch.empty((M,), dtype=torch.int32, device=dev)
        ms = _timed(lambda: p4q.p4q_swiglu_quant_expanded(G, U, Xq, s, Xu, su), a.reps, dev)
        nbytes = 4 * M * K + 3 * M * K // 2 + 8 * M
        print(f"swiglu {M}x{K} of {LD}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "rmsnorm":
        M, K = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        X = (torch.randn((M, K), generator=g, device=dev) * 2.0).to(torch.float16)
        w = (1.0 + 0.2 * torch.randn((K,), generator=g, device=dev)).to(torch.float16)
        Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((M,), dtype=torch.float32, device=dev)
        Xu = torch.empty((M, K), dtype=torch.uint8, device=dev)
        su = torch.empty((M,), dtype=torch.int32, device=dev)
        ms = _timed(lambda: p4q.p4q_rmsnorm_quant_expanded(X, w, 1e-6, Xq, s, Xu, su), a.reps, dev)
        nbytes = 2 * M * K + 2 * K + 3 * M * K // 2 + 8 * M
        print(f"rmsnorm {M}x{K}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "attn":
        B, M, H = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        qkv = torch.randn((B * M, 3 * H * 128), generator=g, device=dev).to(torch.float16)
        Q, K, V = qkv[:, :H * 128], qkv[:, H * 128:2 * H * 128], qkv[:, 2 * H * 128:]
        O = torch.empty((B * M, H * 128), dtype=torch.float16, device=dev)
        ms = _timed(lambda: p4q.p4q_causal_attention(Q, K, V, O, B, M, H, H), a.reps, dev)
        flops = 2 * 2 * 128 * M * (M + 1) / 2 * B * H
        nbytes = 4 * B * M * H * 128 * 2
        print(f"attn {B}x{M} H={H}: {ms * 1e3:.1f} us/call, {flops / ms / 1e9:.1f} TFLOP/s, "
              f"{nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "mse":
        B, M, D = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        Yq = torch.randn((B * M, D), generator=g, device=dev).to(torch.float16)
        Yf = torch.randn((B * M, D), generator=g, device=dev).to(torch.float16)
        e = torch.empty((B,), dtype=torch.float32, device=dev)
        L = torch.empty((1,), dtype=torch.float32, device=dev)
        ws = torch.empty((p4q.p4q_block_mse_workspace_bytes(B),), dtype=torch.uint8, device=dev)
        off = [n * M for n in range(B + 1)]
        ms = _timed(lambda: p4q.p4q_block_mse(Yq, Yf, off, e, L, ws), a.reps, dev)
        nbytes = 4 * B * M * D
        print(f"mse {B}x{M}x{D}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    elif a.case == "topk":
        B, N, K = (int(x) for x in a.args)
        g = torch.Generator(device=dev).manual_seed(0)
        s1 = torch.randn((B, N), generator=g, device=dev)
        s2 = torch.randn((B, N), generator=g, device=dev)
        inter = torch.empty((B,), dtype=torch.int32, device=dev)
        rho = torch.empty((B,), dtype=torch.float32, device=dev)
        ms = _timed(lambda: p4q.p4q_topk_replacement(s1, s2, K, inter, rho), a.reps, dev)
        print(f"topk {B}x{N} K={K}: {ms * 1e3:.1f} us/call, {8 * B * N / ms / 1e6:.1f} GB/s")
    elif a.case == "sweep":
        _sweep(a.args[0], a.reps, dev)
    elif a.case == "hostlink":
        # the host link the end-to-end path copies over: pinned host <-> device, each direction alone and both at once
        nbytes = int(a.args[0]) << 20
        h_in = torch.empty((nbytes,), dtype=torch.uint8).pin_memory()
        h_out = torch.empty((nbytes,), dtype=torch.uint8).pin_memory()
        d_in = torch.empty((nbytes,), dtype=torch.uint8, device=dev)
        d_out = torch.empty((nbytes,), dtype=torch.uint8, device=dev)
        s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)

        def run(h2d, d2h):
            torch.cuda.synchronize()
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record()
            s_in.wait_event(a0)
            s_out.wait_event(a0)
            if h2d:
                with torch.cuda.stream(s_in):
                    d_in.copy_(h_in, non_blocking=True)
            if d2h:
                with torch.cuda.stream(s_out):
                    h_out.copy_(d_out, non_blocking=True)
            torch.cuda.current_stream().wait_stream(s_in)
            torch.cuda.current_stream().wait_stream(s_out)
            a1.record()
            torch.cuda.synchronize()
            return a0.elapsed_time(a1)

        for name, h2d, d2h in (("host->device", True, False), ("device->host", False, True), ("both at once", True, True)):
            ms = min(run(h2d, d2h) for _ in range(max(a.reps, 2)))
            print(f"hostlink {name} {nbytes >> 20} MiB each: {ms * 1e3:.1f} us, {nbytes / ms / 1e6:.1f} GB/s per direction")
    elif a.case == "peak":
        kind, iters = a.args[0], int(a.args[1])
        sink = torch.zeros((8192,), dtype=torch.int32, device=dev)
        ops = p4q.p4q_peak_probe(kind, iters, sink)
        ms = _timed(lambda: p4q.p4q_peak_probe(kind, iters, sink), a.reps, dev)
        print(f"peak {kind} x{iters}: {ms * 1e3:.1f} us/call, {ops / ms / 1e9:.1f} TOPS")
    elif a.case == "saliency":
        B, N = (int(x) for x in a.args)
        v = wl.vision_attention(B, N, seed=0)
        q, kc, k = (torch.from_numpy(t).to(dev) for t in (v.q_cls, v.k_cls, v.k))
        A = torch.empty((B, N), dtype=torch.float32, device=dev)
        ms = _timed(lambda: p4q.p4q_cls_saliency(q, kc, k, A), a.reps, dev)
        nbytes = 2 * (q.numel() + kc.numel() + k.numel()) + 4 * A.numel()
        print(f"saliency {B}x{N}: {ms * 1e3:.1f} us/call, {nbytes / ms / 1e6:.1f} GB/s")
    else:
        w = wl.WORKLOADS[a.args[0]]
        if len(a.args) > 1:  # the same workload on fewer (or more) images
            w = dataclasses.replace(w, B=int(a.args[1]))
        x = wl.selector_inputs(w)
        V, Q, A, T = (torch.from_numpy(t).to(dev) for t in (x.V, x.Q, x.A, x.text))
        ws = p4q.select_workspace(w.B, w.N, w.d, w.J, w.K, dev)
        idx = torch.empty((w.B, w.K), dtype=torch.int32, device=dev)
        X = torch.empty((w.B, w.K + w.T, w.d), dtype=torch.float16, device=dev)
        Xq = torch.empty((w.M, w.d // 2), dtype=torch.uint8, device=dev)
        s = torch.empty((w.M,), dtype=torch.float32, device=dev)
        ms = _timed(lambda: p4q.p4q_select_gather_quant(V, Q, A, T, w.K, idx, X, Xq, s, ws), a.reps, dev)
        print(f"select {w.name}: {ms * 1e3:.1f} us/call, {ms * 1e3 / w.B:.2f} us/image")
    return 0


if __name__ == "__main__":
    sys.exit(main())

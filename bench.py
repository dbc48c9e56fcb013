"""Benchmark of the P4Q pruned W4A4 hot path on GB300.

One step = the whole path over one batch of the LLaVA-NeXT-13B-shaped workload
(32 images x 2880 visual tokens of 5120 fp16 features, heavy-tailed outlier
channels, + 64 text tokens each, budget 640 kept tokens per image; the
largest of the LLaVA-shaped workloads, and one GPU holds it):
  p4q_select_gather_quant  fake-quant -> query / saliency / diversity stages
                           -> gather of the kept FP16 rows + text -> INT4
  (the selector's gather and the two re-quantizations also write their
  codes in the expanded form, one byte per code, that the GEMMs read)
  p4q_expand_codes         each GEMM's packed INT4 weights, per call, into
                           that GEMM's scratch, on a side stream from the
                           start of the step
  p4q_w4a4_linear_expanded x 3  q|k|v|gate|up (one GEMM over the
                           concatenated output channels) on the pruned
                           sequence (M = 22528), o on the re-quantized q
                           output, down on the re-quantized up output
                           (2 x p4q_quant_act_expanded on column blocks;
                           the o chain on a third stream beside the
                           down chain).
The metric is W4A4 linear TOPS: 2 * M * N * K integer ops of the seven linears
per step divided by the step time (the selector's time included); the
selector's share is also reported as microseconds per image.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {p4q,reference}]
                  [--workload NAME]

--workload runs the same step on another of the LLaVA-shaped workloads (the
one-image 576-token case, the 8 x 576-token LLaVA-1.5-7B batch, the
16 x 2880-token LLaVA-NeXT-7B batch over 32 decoder layers); the default is
the 32-image batch above.

--impl reference times the CPU oracle (test infrastructure) on a bounded
sample of the same workload. Under torchrun each rank runs its own batch
(weak scaling, no collective on the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2609_34867_gb300 import workloads as wl  # noqa: E402

METRIC = "W4A4 prefill linear TOPS (% INT8 tensor peak); select+prune µs/image"
WORKLOAD = wl.LLAVANEXT_13B
FLUSH_BYTES = 512 << 20  # > 129 MB L2, written and then read between timed steps

# Latest ncu capture of the dominant kernel (the expanded-operand GEMM): mean
# DRAM bytes (read + write) per launch over the three GEMM shapes of one step
# of the 32 x 2880 x 5120 workload (22528 x 43008 x 5120, 22528 x 5120 x 5120,
# 22528 x 5120 x 13824), valid only while the GEMM source is unchanged since
# the capture.
PROFILED_GEMM = {"source_sha1": "9e6ce95c71d8db37f51a4c972b54b5a399a2ce4a", "dram_bytes_per_launch": 1806128981}


def gemm_source_sha1() -> str:
    p = os.path.join(ROOT, "paper_2609_34867_gb300", "csrc", "p4q_gemm8.cu")
    return hashlib.sha1(open(p, "rb").read()).hexdigest()


def linear_ops(w: wl.Workload) -> int:
    return w.layers * sum(2 * w.M * l.n_out * l.k_in for l in w.linears)


def rank_seed(w: wl.Workload, rank: int) -> int:
    """Input seed of a rank's batch: every rank draws its own images and text
    (weights are replicated: they depend on the workload and layer only)."""
    return w.seed + rank


def max_over_ranks(values, world: int, device):
    """Element-wise maximum of per-rank timings over all ranks (all_reduce MAX;
    the identity for a single process). The job takes as long as its slowest
    rank."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def whole_job_tops(ops_per_rank: int, world: int, ms_per_step: float) -> float:
    """Aggregate throughput: the integer ops of every rank's batch over the
    (max-over-ranks) step time."""
    return ops_per_rank * world / (ms_per_step * 1e-3) / 1e12


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        return None


def fp8_peak_tops(sustained: bool):
    """Dense FP8 tensor peak derived from the measured bf16 cuBLAS rate: x the
    nominal fp8 / bf16 ratio (4.5 / 2.25). Reported beside the FP8 rate this
    run measures itself (p4q_peak_probe), which is the roofline's peak."""
    pk = measured_peaks()
    if pk:
        bf = pk.get("bf16_tflops_sustained" if sustained else "bf16_tflops")
        return 2.0 * bf, ("measured bf16 %s x 2 (nominal fp8/bf16 ratio), MEASURED_PEAKS.json"
                          % ("sustained" if sustained else "burst"))
    return 2.0 * (1700.0 if sustained else 1900.0), "fallback bf16 x 2"


def hbm_peak_gbs():
    pk = measured_peaks()
    if pk and pk.get("hbm_gbs"):
        return float(pk["hbm_gbs"]), "measured copy, MEASURED_PEAKS.json"
    return 6800.0, "fallback 6.8 TB/s"


def select_budget(w: wl.Workload):
    """(K_q, K_s, K_d) of Sec. 3.2's split in integers (concepts and CLS
    saliency present in every bench workload)."""
    kq = 300 * w.K // 1000
    ks = 200 * w.K // 1000
    return kq, ks, w.K - kq - ks


def selector_roofline(w: wl.Workload, us_per_image: float, hbm_gbs: float, f8_tops: float) -> dict:
    """Select + prune per image against the larger of its two bounds:
    - HBM: one read of the image's features, its text rows and its kept rows
      (the gather), and the codes of the pruned sequence written:
      (N d 2 + T d 2 + K d 2 + (K + T)(d / 2 + 4)) bytes at the measured copy
      bandwidth;
    - diversity MACs on the FP8 tensor pipe: (K_q + K_s) N d for the initial
      maxima plus sum over the K_d greedy rounds of the free tokens' d-long
      dot products, 2 ops each, at the FP8 rate measured in this run."""
    kq, ks, kd = select_budget(w)
    nbytes = w.N * w.d * 2 + w.T * w.d * 2 + w.K * w.d * 2 + (w.K + w.T) * (w.d // 2 + 4)
    macs = (kq + ks) * w.N * w.d + sum((w.N - kq - ks - t) * w.d for t in range(kd))
    hbm_us = nbytes / (hbm_gbs * 1e3)
    mac_us = 2.0 * macs / (f8_tops * 1e6)
    bound = max(hbm_us, mac_us)
    return {"bound": "hbm" if hbm_us >= mac_us else "tensor", "achieved_us_per_image": round(us_per_image, 3),
            "bound_us_per_image": round(bound, 3), "frac": round(bound / us_per_image, 4),
            "hbm_bytes_per_image": int(nbytes), "hbm_us_per_image": round(hbm_us, 3),
            "diversity_macs_per_image": int(macs), "diversity_us_per_image": round(mac_us, 3)}


# --------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"p4q_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        os.remove(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        return {"sm_mhz": float(np.median([r[0] for r in rows])), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------- GPU arm
class L2Flush:
    """Evicts the step's data from the 129 MB L2 before a timed step: writes
    one buffer larger than L2, then reads another, so that L2 holds only clean
    lines of the second buffer and the timed step pays for no write-back of
    the flush."""

    def __init__(self, dev):
        import torch
        self.w = torch.empty((FLUSH_BYTES,), dtype=torch.uint8, device=dev)
        self.r = torch.ones((FLUSH_BYTES // 4,), dtype=torch.float32, device=dev)

    def __call__(self):
        self.w.zero_()
        self.r.amax()


class Step:
    """Device buffers and weights of one rank, and the step itself.

    The inputs are drawn with `seed`; the weights of decoder layer l with
    wl.weight_seed(w.seed + l, linear id), the same on every rank (replicated
    weights, independent batches). Every layer runs on the pruned sequence:
    q, k, v, gate, up on its INT4 codes, o on the re-quantized q output, down
    on the re-quantized up output. Linears that read the same input run as one
    GEMM over their concatenated output channels (q|k|v|gate|up), which
    computes exactly the same outputs (the weight quantizer works per output
    channel) with fewer launches and fuller waves of tiles: 1072 tiles of
    256 x 256 take 15 rounds of the 76 CTA pairs, where q|k|v and gate|up
    apart take 6 + 10."""

    FUSE = (("qkv_gate_up", ("q", "k", "v", "gate", "up")),)
    REQUANT = {"o": "q", "down": "up"}  # linear -> the linear whose output it re-quantizes

    def __init__(self, w: wl.Workload, dev, seed: int):
        import torch
        from paper_2609_34867_gb300 import p4q
        self.torch, self.p4q, self.w, self.dev = torch, p4q, w, dev
        x = wl.selector_inputs(w, seed=seed)
        self.host = {"V": x.V, "Q": x.Q, "A": x.A, "text": x.text}
        self.V = torch.from_numpy(x.V).to(dev)
        self.Q = torch.from_numpy(x.Q).to(dev)
        self.A = torch.from_numpy(x.A).to(dev)
        self.text = torch.from_numpy(x.text).to(dev)
        B, N, d, K, T = w.B, w.N, w.d, w.K, w.T
        self.ws = p4q.select_workspace(B, N, d, w.J, K, dev)
        self.idx = torch.empty((B, K), dtype=torch.int32, device=dev)
        self.X = torch.empty((B, K + T, d), dtype=torch.float16, device=dev)
        M = w.M
        self.Xq = torch.empty((M, d // 2), dtype=torch.uint8, device=dev)
        self.s_a = torch.empty((M,), dtype=torch.float32, device=dev)
        dims = {l.name: l for l in w.linears}
        lid = {l.name: i for i, l in enumerate(w.linears)}
        # GEMMs: fused groups whose members all exist and share k_in, else single linears
        self.gemms, taken = [], set()
        for gname, members in self.FUSE:
            if all(m in dims for m in members) and len({dims[m].k_in for m in members}) == 1:
                self.gemms.append((gname, members))
                taken.update(members)
        for l in w.linears:
            if l.name not in taken:
                self.gemms.append((l.name, (l.name,)))
        self.col = {}  # linear -> (gemm, first output column, width)
        for gname, members in self.gemms:
            off = 0
            for m in members:
                self.col[m] = (gname, off, dims[m].n_out)
                off += dims[m].n_out
        self.Wq, self.s_w, self.Y = {}, {}, {}
        for gname, members in self.gemms:
            n_out = sum(dims[m].n_out for m in members)
            self.Y[gname] = torch.empty((M, n_out), dtype=torch.float16, device=dev)
            for layer in range(w.layers):
                W = torch.cat([torch.from_numpy(wl.weight(dims[m].k_in, dims[m].n_out,
                                                          wl.weight_seed(w.seed + layer, lid[m]))) for m in members])
                self.Wq[layer, gname], self.s_w[layer, gname] = p4q.quant_weight(W.to(dev))
                del W
        self.Xq_re, self.s_re = {}, {}
        for name, src in self.REQUANT.items():
            if name in dims:
                assert src in dims, f"{name} needs the {src} linear"
                self.Xq_re[name] = torch.empty((M, dims[name].k_in // 2), dtype=torch.uint8, device=dev)
                self.s_re[name] = torch.empty((M,), dtype=torch.float32, device=dev)
        self.out_name = w.linears[-1].name
        # Expanded operands (one byte per code + row sums, p4q_expand_codes):
        # the pruned sequence once per step for every GEMM that reads it, the
        # re-quantized o / down inputs, and each GEMM's weights per call into
        # one scratch (the weights stay packed INT4 in memory).
        self.Xu = torch.empty((M, d), dtype=torch.uint8, device=dev)
        self.sXu = torch.empty((M,), dtype=torch.int32, device=dev)
        self.Xu_re, self.sXu_re = {}, {}
        for name in self.Xq_re:
            self.Xu_re[name] = torch.empty((M, dims[name].k_in), dtype=torch.uint8, device=dev)
            self.sXu_re[name] = torch.empty((M,), dtype=torch.int32, device=dev)
        # When every re-quantized block is a column block of one GEMM's output,
        # that GEMM records each row's abs-max per block (its row-max epilogue)
        # and each block is quantized in one streaming pass
        # (p4q_quant_act_expanded_rowmax) instead of two.
        srcs = {self.col[self.REQUANT[n]][0] for n in self.Xq_re}
        self.rm_gemm = None
        if len(srcs) == 1 and 1 <= len(self.Xq_re) <= 2:
            names = sorted(self.Xq_re, key=lambda n: self.col[self.REQUANT[n]][1])
            blocks = [tuple(self.col[self.REQUANT[n]][1:]) for n in names]
            if all(off % 32 == 0 and n % 256 == 0 for off, n in blocks):
                self.rm_gemm, self.rm_names, self.rm_blocks = srcs.pop(), names, blocks
                self.rowmax = torch.empty((len(names), M), dtype=torch.int32, device=dev)
        # the one-pass re-quantization writes only the expanded codes the next
        # GEMM reads (no packed copy: nothing in the step reads it)
        self.packed_requant = self.rm_gemm is None
        # one weight scratch per GEMM of a layer: the weights expand on a side
        # stream, ahead of the GEMMs that read them (see body)
        self.slot = {g: i for i, (g, _) in enumerate(self.gemms)}
        self.Wu = [torch.empty((self.Wq[0, g].shape[0], self.Wq[0, g].shape[1] * 2), dtype=torch.uint8, device=dev)
                   for g, _ in self.gemms]
        self.sWu = [torch.empty((self.Wq[0, g].shape[0],), dtype=torch.int32, device=dev) for g, _ in self.gemms]
        self.side = torch.cuda.Stream(device=dev)
        self.aux = torch.cuda.Stream(device=dev)
        # The step is a chain of segments (selector, each expansion, each GEMM,
        # each re-quantization); the timed loop replays it as one CUDA graph,
        # the breakdown replays one graph per segment with events between them.
        self.segments = [("select", "select", self._select)]
        self.gemm_calls = []  # (layer, gemm, input) in step order
        for layer in range(w.layers):
            for gname, members in self.gemms:
                if members[0] in self.REQUANT:
                    name = members[0]
                    self.segments.append(("quant", "quant_" + name, (lambda n=name: self._requant(n))))
                    xin = (lambda n=name: (self.Xu_re[n], self.sXu_re[n], self.s_re[n]))
                else:
                    xin = (lambda: (self.Xu, self.sXu, self.s_a))
                self.segments.append(("expand", "expand_w_" + gname, (lambda l=layer, g=gname: self._expand_w(l, g))))
                self.segments.append(("linear", gname, (lambda l=layer, g=gname, x=xin: self._gemm(l, g, *x()))))
                self.gemm_calls.append((layer, gname, xin))
        self.lin_ops = {g: sum(2 * w.M * dims[m].n_out * dims[m].k_in for m in members) * w.layers
                        for g, members in self.gemms}
        self.graphs = None
        self.launches_per_step = None
        self.events = [torch.cuda.Event(enable_timing=True) for _ in range(len(self.segments) + 1)]

    def output(self, name):
        """The [M, n_out] output of one linear (a column block of its GEMM's output)."""
        g, off, n = self.col[name]
        return self.Y[g][:, off:off + n]

    def weight(self, layer, name):
        """The packed INT4 rows and scales of one linear inside its GEMM's weight."""
        g, off, n = self.col[name]
        return self.Wq[layer, g][off:off + n], self.s_w[layer, g][off:off + n]

    def _select(self):
        # the pruned sequence's expanded codes only: the GEMMs read them, nothing reads a packed copy
        self.p4q.p4q_select_gather_quant_expanded(self.V, self.Q, self.A, self.text, self.w.K, self.idx, self.X,
                                                  None, self.s_a, self.Xu, self.sXu, self.ws)

    def _expand_w(self, layer, gname, stream=None):
        k = self.slot[gname]
        self.p4q.p4q_expand_codes(self.Wq[layer, gname], self.Wu[k], self.sWu[k], stream)

    def _gemm(self, layer, gname, Xu, sXu, s, stream=None):
        k = self.slot[gname]
        if gname == self.rm_gemm:
            self.p4q.p4q_w4a4_linear_expanded_rowmax(Xu, sXu, s, self.Wu[k], self.sWu[k], self.s_w[layer, gname],
                                                     self.Y[gname], self.rm_blocks, self.rowmax, stream)
        else:
            self.p4q.p4q_w4a4_linear_expanded(Xu, sXu, s, self.Wu[k], self.sWu[k], self.s_w[layer, gname],
                                              self.Y[gname], stream)

    def _requant(self, name, stream=None):
        """The per-token codes of the block of the source GEMM's output that
        linear `name` reads (R10): one pass with the row maxima the GEMM
        recorded, else the two-pass quantizer."""
        if self.rm_gemm is None:
            self.p4q.p4q_quant_act_expanded(self.output(self.REQUANT[name]), self.Xq_re[name], self.s_re[name],
                                            self.Xu_re[name], self.sXu_re[name], stream)
            return
        b = self.rm_names.index(name)
        self.p4q.p4q_quant_act_expanded_rowmax(self.Y[self.rm_gemm], [self.rm_blocks[b]], self.rowmax[b:b + 1],
                                               None, [self.s_re[name]], [self.Xu_re[name]], [self.sXu_re[name]],
                                               stream)

    def body_serial(self):
        """The step's segments one after another on the current stream."""
        for _, _, fn in self.segments:
            fn()

    def body(self, out_free=None):
        """The step as plain C-ABI calls (no graph), on three streams:
        - side: every GEMM's weight expansion, into that GEMM's scratch, in
          step order (a later layer's waits until the previous layer's GEMM
          has read the scratch). The first GEMM of a layer has its weights
          expanded ahead (beside the selector, or beside the previous
          layer's GEMMs); the layer's other GEMMs have theirs expanded once
          that first GEMM is about to start, so the expansion streams beside
          a tensor-bound GEMM instead of competing with the memory-bound
          selector for HBM;
        - aux: the o chain (re-quantization of the q block, o GEMM), beside
          the down chain (re-quantization of the up block, down GEMM);
        - the current stream: everything else.
        out_free: an event the GEMM that writes the step's output waits for
        (a copy of the previous step's output still reading it)."""
        torch = self.torch
        main = torch.cuda.current_stream()
        self.side.wait_stream(main)  # fork: the inputs of this step are in place
        self.aux.wait_stream(main)
        n = len(self.gemm_calls)
        ngemm = len(self.gemms)
        ready = [torch.cuda.Event() for _ in range(n)]
        freed = [torch.cuda.Event() for _ in range(n)]

        def expand(i, after=None):
            """Call i's weights into its GEMM's scratch, on the side stream."""
            layer, gname, _ = self.gemm_calls[i]
            with torch.cuda.stream(self.side):
                if i >= ngemm:
                    self.side.wait_event(freed[i - ngemm])
                if after is not None:
                    self.side.wait_event(after)
                self._expand_w(layer, gname, self.side)
                ready[i].record(self.side)

        expand(0)
        self._select()
        members = dict(self.gemms)
        o_src = self.col[self.REQUANT["o"]][0] if "o" in self.Xq_re else None
        src_done, o_read = None, None
        for i, (layer, gname, xin) in enumerate(self.gemm_calls):
            first = members[gname][0]
            if i % ngemm == 0:
                # the layer's first GEMM is next: its other GEMMs' weights now
                go = torch.cuda.Event()
                go.record(main)
                for j in range(i + 1, i + ngemm):
                    expand(j, go)
            if first == "o":
                with torch.cuda.stream(self.aux):
                    if src_done is not None:
                        self.aux.wait_event(src_done)
                    self._requant("o", self.aux)
                    o_read = torch.cuda.Event()
                    o_read.record(self.aux)
                    self.aux.wait_event(ready[i])
                    self._gemm(layer, gname, *xin(), self.aux)
                    freed[i].record(self.aux)
                continue
            if first in self.REQUANT:
                self._requant(first)
            if gname == o_src and o_read is not None:
                main.wait_event(o_read)  # the previous layer's o chain has read this GEMM's output
            if out_free is not None and self.out_name in members[gname]:
                main.wait_event(out_free)
            main.wait_event(ready[i])
            self._gemm(layer, gname, *xin())
            freed[i].record(main)
            if i % ngemm == 0 and i + ngemm < n:
                expand(i + ngemm)  # the next layer's first GEMM, once this one has read the scratch
            if gname == o_src:
                src_done = torch.cuda.Event()
                src_done.record(main)
        main.wait_stream(self.side)  # join
        main.wait_stream(self.aux)

    def capture(self):
        """Captures the whole step into one CUDA graph (consecutive kernels
        overlap their launch and set-up with the previous kernel's tail), and
        every segment into its own graph for per-segment timing (after warm-up
        calls have set up the kernels' attributes). Garbage collection is
        done before and held off during the captures: a collected object that
        owns a CUDA graph (a Step lives in a reference cycle through its
        segment closures) would destroy it mid-capture, which invalidates the
        capture."""
        import gc
        torch = self.torch
        gc.collect()
        was_enabled = gc.isenabled()
        gc.disable()
        try:
            self.graphs = []
            for _, _, fn in self.segments:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    fn()
                self.graphs.append(g)
            self.body()  # warm the side-stream path before capturing it
            torch.cuda.synchronize()
            n0 = self.p4q.p4q_launch_count()
            self.full = torch.cuda.CUDAGraph()
            with torch.cuda.graph(self.full):
                self.body()
            self.launches_per_step = self.p4q.p4q_launch_count() - n0
        finally:
            if was_enabled:
                gc.enable()

    def __call__(self, segments: bool = False):
        """One step: the whole-step graph, or (segments=True) the segment
        graphs with events between them (see kernel_times)."""
        if self.graphs is None:
            self.body()
            return
        if not segments:
            self.full.replay()
            return
        self.events[0].record()
        for i, g in enumerate(self.graphs):
            g.replay()
            self.events[i + 1].record()

    def kernel_times(self):
        """Milliseconds of the most recent graph step (after a sync):
        {"select": ms, "quant": ms summed, "linear": {gemm: ms summed over layers}}."""
        out = {"select": 0.0, "quant": 0.0, "expand": 0.0, "linear": {g: 0.0 for g, _ in self.gemms}}
        for i, (kind, name, _) in enumerate(self.segments):
            ms = self.events[i].elapsed_time(self.events[i + 1])
            if kind == "linear":
                out["linear"][name] += ms
            else:
                out[kind] += ms
        return out


def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    from paper_2609_34867_gb300 import build as _build
    from paper_2609_34867_gb300 import p4q
    if rank == 0 or not os.path.exists(_build.LIB):
        _build.build()
    if world > 1:
        dist.barrier()
    p4q.lib()
    w = wl.WORKLOADS[args.workload]
    step = Step(w, dev, seed=rank_seed(w, rank))
    flush = L2Flush(dev)
    for _ in range(args.warmup):
        flush()
        step()
    torch.cuda.synchronize()
    if p4q.p4q_device_status() != 0:
        raise RuntimeError("device status not ok after warm-up")
    step.capture()
    for _ in range(3):
        flush()
        step()
    torch.cuda.synchronize()
    # the pipes' own rates on this GPU (untimed region): the roofline's FP8
    # peak and the s8 basis of the metric's "% INT8 tensor peak"
    from paper_2609_34867_gb300 import kernel_cases as kc
    f8_tops = kc.peak_tops("f8", dev)
    s8_tops = kc.peak_tops("s8", dev)

    # ---- device-timed region: K graph replays, L2 flushed before each, events
    # around each replay; per-kernel times from the events inside the graph
    clocks = ClockSampler(int(os.environ.get("P4Q_NVSMI_INDEX", local_rank)))
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    step_ms, sel_ms, exp_ms, quant_ms, gemm_ms = [], [], [], [], {g: [] for g, _ in step.gemms}
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush()
        e_start.record()
        step()
        e_end.record()
        torch.cuda.synchronize()
        step_ms.append(e_start.elapsed_time(e_end))
    t_wall = time.perf_counter() - t_wall
    # per-segment times (selector, each GEMM) from the segment graphs
    for i in range(min(args.steps, 200)):
        flush()
        step(segments=True)
        torch.cuda.synchronize()
        kt = step.kernel_times()
        sel_ms.append(kt["select"])
        exp_ms.append(kt["expand"])
        quant_ms.append(kt["quant"])
        for n in gemm_ms:
            gemm_ms[n].append(kt["linear"][n])
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    launches = step.launches_per_step * args.steps
    if p4q.p4q_device_status() != 0:
        raise RuntimeError("device status not ok after the timed region")
    total_ms = float(np.sum(step_ms))
    sel_ms = np.array(sel_ms)
    gemm_ops = float(sum(step.lin_ops.values()))
    gemm_time_ms = float(sum(np.mean(v) for v in gemm_ms.values()))

    # ---- end to end through the C ABI with host buffers (pinned), copies timed
    e2e_ms = None
    h2d_bytes = d2h_bytes = 0
    if args.e2e_steps > 0:
        hostV = torch.from_numpy(step.host["V"]).pin_memory()
        hostQ = torch.from_numpy(step.host["Q"]).pin_memory()
        hostA = torch.from_numpy(step.host["A"]).pin_memory()
        hostT = torch.from_numpy(step.host["text"]).pin_memory()
        outY = torch.empty(step.output(step.out_name).shape, dtype=torch.float16).pin_memory()
        outI = torch.empty(step.idx.shape, dtype=torch.int32).pin_memory()
        h2d_bytes = sum(t.numel() * t.element_size() for t in (hostV, hostQ, hostA, hostT))
        d2h_bytes = outY.numel() * 2 + outI.numel() * 4
        # one step at a time: copies in, the step, copies out, nothing overlapped
        times = []
        for i in range(min(args.e2e_steps, 10) + 2):
            flush()
            torch.cuda.synchronize()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            step.V.copy_(hostV, non_blocking=True)
            step.Q.copy_(hostQ, non_blocking=True)
            step.A.copy_(hostA, non_blocking=True)
            step.text.copy_(hostT, non_blocking=True)
            step.body()  # the C-ABI calls themselves, no graph
            outY.copy_(step.output(step.out_name), non_blocking=True)
            outI.copy_(step.idx, non_blocking=True)
            b.record()
            torch.cuda.synchronize()
            if i >= 2:
                times.append(a.elapsed_time(b))
        e2e_serial_ms = float(np.mean(times))
        # a stream of batches: while step i computes, one copy stream brings in
        # the inputs of step i + 1 (two device input sets, alternating) and
        # another copies out the result of step i - 1 (the host link carries
        # both directions at once); every step still copies its own inputs in
        # from pinned host memory and its result out. No L2 flush between
        # steps: each step moves more than the L2 holds (V, the packed weights
        # and their expanded copies).
        main = torch.cuda.current_stream()
        copy = torch.cuda.Stream(device=dev)      # host -> device
        copy_out = torch.cuda.Stream(device=dev)  # device -> host
        sets = [(step.V, step.Q, step.A, step.text, step.idx),
                tuple(torch.empty_like(t) for t in (step.V, step.Q, step.A, step.text, step.idx))]
        outYs = [outY, torch.empty_like(outY).pin_memory()]
        outIs = [outI, torch.empty_like(outI).pin_memory()]
        E = args.e2e_steps
        in_ready = [torch.cuda.Event() for _ in range(E + 1)]
        done = [torch.cuda.Event() for _ in range(E)]
        copied = [torch.cuda.Event() for _ in range(E)]

        def h2d(i):
            V, Q, A, T, _ = sets[i % 2]
            with torch.cuda.stream(copy):
                if i >= 2:
                    copy.wait_event(done[i - 2])  # step i - 2 has finished with this set
                V.copy_(hostV, non_blocking=True)
                Q.copy_(hostQ, non_blocking=True)
                A.copy_(hostA, non_blocking=True)
                T.copy_(hostT, non_blocking=True)
                in_ready[i].record(copy)

        for rep_ in range(2):  # the first pass warms the path, the second is timed
            torch.cuda.synchronize()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            t_host = time.perf_counter()
            a.record(main)
            copy.wait_event(a)
            copy_out.wait_event(a)
            h2d(0)
            for i in range(E):
                if i + 1 < E:
                    h2d(i + 1)
                main.wait_event(in_ready[i])
                if i >= 2:
                    main.wait_event(copied[i - 2])  # the result copy of step i - 2 has read its idx set
                step.V, step.Q, step.A, step.text, step.idx = sets[i % 2]
                step.body(out_free=copied[i - 1] if i >= 1 else None)
                done[i].record(main)
                with torch.cuda.stream(copy_out):
                    copy_out.wait_event(done[i])
                    outYs[i % 2].copy_(step.output(step.out_name), non_blocking=True)
                    outIs[i % 2].copy_(step.idx, non_blocking=True)
                    copied[i].record(copy_out)
            main.wait_stream(copy)
            main.wait_stream(copy_out)
            b.record(main)
            host_ms = (time.perf_counter() - t_host) * 1e3 / E  # enqueueing only: nothing waited on yet
            torch.cuda.synchronize()
        step.V, step.Q, step.A, step.text, step.idx = sets[0]
        e2e_ms = a.elapsed_time(b) / E
        e2e_host_ms = host_ms
        # every step had the same inputs and the kernels are deterministic: the
        # two result buffers must agree bit for bit (a race in the overlap would not)
        if E >= 2 and not (torch.equal(outYs[0], outYs[1]) and torch.equal(outIs[0], outIs[1])):
            raise RuntimeError("pipelined end-to-end steps disagree: an overlap race")

    # ---- reduce over ranks (max time)
    total_ms, e2e_max = max_over_ranks([total_ms, e2e_ms or 0.0], world, dev)
    if rank != 0:
        return None

    ops = linear_ops(w)
    ms_per_step = total_ms / args.steps
    value = whole_job_tops(ops, world, ms_per_step)
    # the roofline's peak: the FP8 MMA-only rate measured above; the bf16-derived
    # figure (burst unless the clocks show the power cap) is reported beside it
    sustained = bool(clk and "sw_power_cap" in clk["reasons"])
    peak_bf, peak_bf_src = fp8_peak_tops(sustained)
    peak = f8_tops
    hbm_gbs, hbm_src = hbm_peak_gbs()
    ach = gemm_ops / (gemm_time_ms * 1e-3) / 1e12
    exp_time_ms = float(np.mean(exp_ms))
    ach_lin = gemm_ops / ((gemm_time_ms + exp_time_ms) * 1e-3) / 1e12
    sel_us = float(sel_ms.mean()) * 1e3 / w.B
    n_gemm = len(step.gemms) * w.layers * args.steps
    traffic = None
    if PROFILED_GEMM["source_sha1"] == gemm_source_sha1():
        traffic = PROFILED_GEMM["dram_bytes_per_launch"]
    rec = {
        "metric": METRIC,
        "value": round(value, 3),
        "unit": "TOPS",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int4",
        "data": "synthetic",
        "config": {
            "workload": w.name, "B": w.B, "N": w.N, "d": w.d, "K": w.K, "T": w.T, "J": w.J, "M": w.M,
            "linears": "; ".join(f"{l.name} {l.k_in}->{l.n_out}" for l in w.linears), "layers": w.layers,
            "gemms": "; ".join(f"{g}={'|'.join(m)}" for g, m in step.gemms),
            "alpha_beta_gamma": "0.3/0.2/0.5", "l2": "flushed before every timed step: 512 MiB written, then another 512 MiB read (no dirty flush lines left to write back inside the timed region)",
            "timing": "CUDA events around each step (one CUDA graph per step), summed over the K steps; "
                      "selector and per-GEMM times from segment graphs with events between them",
            "parallelism": f"dp{world} (independent batches)"},
        "select_prune_us_per_image": round(sel_us, 3),
        "select_prune_roofline": selector_roofline(w, sel_us, hbm_gbs, f8_tops),
        "expand_us_per_step": round(exp_time_ms * 1e3, 2),
        "requant_us_per_step": round(float(np.mean(quant_ms)) * 1e3, 2),
        "gemm_tops": round(ach, 3),
        "pct_int8_tensor_peak": round(100.0 * ach / s8_tops, 2),
        "pct_int8_tensor_peak_basis": "mma.sync m16n8k32 s8 x s8 -> s32 loop measured in this run "
                                      "(p4q_peak_probe kind 1): %.1f TOPS" % s8_tops,
        "pct_fp8_tensor_peak": round(100.0 * ach / peak, 2),
        "peaks_measured": {"f8_tcgen05_tops": round(f8_tops, 1), "s8_mma_sync_tops": round(s8_tops, 1),
                           "fp8_from_bf16_tops": round(peak_bf, 1), "fp8_from_bf16_source": peak_bf_src,
                           "hbm_gbs": hbm_gbs, "hbm_source": hbm_src},
        "linear_incl_expand": {"achieved": round(ach_lin, 3), "unit": "TFLOP/s", "frac": round(ach_lin / peak, 4),
                               "note": "the GEMM kernels' time plus the per-call expansion of their packed "
                                       "INT4 weights (p4q_expand_codes), as if not overlapped"},
        "roofline": {"bound": "tensor", "kernel": "w4a4_gemm8_pair_kernel (tcgen05 kind::f8f6f4, cta_group::2, TMA-fed expanded operands)",
                     "achieved": round(ach, 3), "peak": round(peak, 1), "unit": "TFLOP/s",
                     "frac": round(ach / peak, 4), "traffic": traffic,
                     "peak_source": "measured in this run: tcgen05 kind::f8f6f4 MMA-only loop on operands in "
                                    "shared memory, 76 CTA pairs (p4q_peak_probe kind 0)",
                     "launches_timed": n_gemm,
                     "note": "integer ops on the FP8 tensor pipe; sm_103a has no integer tcgen05 MMA kind",
                     "per_gemm_us": {n: round(float(np.mean(v)) * 1e3, 2) for n, v in gemm_ms.items()}},
        "gpu_launches": int(launches),
        "launch": "1 CUDA graph replay per step (%d kernels of libp4q per step, programmatic dependent launch)" % (
            step.launches_per_step),
        "clocks": clk,
    }
    if e2e_ms is not None:
        rec["e2e"] = {"value": round(whole_job_tops(ops, world, e2e_max), 3), "unit": "TOPS",
                      "h2d_bytes_per_step": int(h2d_bytes), "d2h_bytes_per_step": int(d2h_bytes),
                      "ms_per_step": round(e2e_max, 4), "steps": args.e2e_steps,
                      "timing": "a stream of steps through the C-ABI calls (no graph): each step's inputs copied in "
                                "from pinned host memory on one copy stream and its result copied out on another, "
                                "overlapping the neighbouring steps' compute; total time / steps, no L2 flush (each "
                                "step moves more than the L2 holds)",
                      "serial_ms_per_step": round(e2e_serial_ms, 4),
                      "host_enqueue_ms_per_step": round(e2e_host_ms, 4),
                      "serial_value": round(whole_job_tops(ops, world, e2e_serial_ms), 3)}
    if not args.no_cpu_baseline and world == 1:
        rec["cpu_baseline"] = cpu_baseline(w, args.cpu_threads)
    return rec


# --------------------------------------------------------------------- CPU oracle
class OracleSampler:
    """Times the CPU oracle on bounded pieces of one step and scales them up.

    Pieces: the selector + gather + quantize of one image (x B images), and each
    of the seven linears on `rows` rows of the pruned sequence (x M / rows),
    with the o and down inputs re-quantized from the q and up outputs as in the
    step. Weight quantization is offline and not timed."""

    def __init__(self, w: wl.Workload, threads: int, rows: int = 4):
        import oracle
        self.o, self.w, self.rows = oracle, w, rows
        self.cores = oracle.set_threads(threads)
        self.x = wl.selector_inputs(w)
        idx = oracle.select_batch(self.x.V[:1], w.K, self.x.Q[:1], self.x.A[:1])
        X = oracle.gather(self.x.V[:1], idx, self.x.text[:1]).reshape(-1, w.d)[:rows]
        self.ca, self.sa = oracle.quantize_rows(X)
        self.cw = {}
        for lid, lin in enumerate(w.linears):
            self.cw[lin.name] = oracle.quantize_rows(wl.weight(lin.k_in, lin.n_out, wl.weight_seed(w.seed, lid)))
        self.y = {n: oracle.linear(self.ca, self.sa, *self.cw[n]) for n in ("q", "up") if n in self.cw}
        self.pieces = [("select", None)] + [("linear", l.name) for l in w.linears]
        self.times = {i: [] for i in range(len(self.pieces))}
        self.image = 0

    def run_piece(self, i: int) -> float:
        o, w = self.o, self.w
        kind, name = self.pieces[i % len(self.pieces)]
        t0 = time.perf_counter()
        if kind == "select":
            b = self.image % w.B
            self.image += 1
            idx = o.select_batch(self.x.V[b:b + 1], w.K, self.x.Q[b:b + 1], self.x.A[b:b + 1])
            o.quantize_rows(o.gather(self.x.V[b:b + 1], idx, self.x.text[b:b + 1]).reshape(-1, w.d))
        elif name in ("o", "down"):
            a, s = o.quantize_rows(self.y["q" if name == "o" else "up"])
            o.linear(a, s, *self.cw[name])
        else:
            o.linear(self.ca, self.sa, *self.cw[name])
        dt = time.perf_counter() - t0
        self.times[i % len(self.pieces)].append(dt)
        return dt

    def estimate(self) -> float:
        """Estimated seconds of one full step from the mean time of each piece."""
        w = self.w
        est = 0.0
        for i, (kind, _) in enumerate(self.pieces):
            if not self.times[i]:
                raise RuntimeError("piece not sampled")
            est += float(np.mean(self.times[i])) * (w.B if kind == "select" else w.layers * w.M / self.rows)
        return est

    def breakdown(self) -> dict:
        """The selector piece's mean time per image and the sampled linears'
        integer-op throughput (their ops over their mean times)."""
        sel, ops, sec = None, 0.0, 0.0
        lin = {l.name: l for l in self.w.linears}
        for i, (kind, name) in enumerate(self.pieces):
            if not self.times[i]:
                continue
            t = float(np.mean(self.times[i]))
            if kind == "select":
                sel = t
            else:
                ops += 2.0 * self.rows * lin[name].k_in * lin[name].n_out
                sec += t
        return {"select_ms_per_image": round(sel * 1e3, 3) if sel is not None else None,
                "linear_gops": round(ops / sec / 1e9, 3) if sec > 0 else None}

    def describe(self) -> str:
        w = self.w
        lay = f" x {w.layers} layers" if w.layers > 1 else ""
        return (f"selector+gather+quantize on 1 of {w.B} images (x{w.B}) and each of the {len(w.linears)} linears "
                f"on {self.rows} of {w.M} rows (x{w.M // self.rows}{lay}), o/down inputs re-quantized; "
                f"weight quantization untimed")


def cpu_baseline(w: wl.Workload, threads: int, reps: int = 2):
    s = OracleSampler(w, threads)
    timed = []
    for _ in range(reps):
        for i in range(len(s.pieces)):
            timed.append(s.run_piece(i))
    est = s.estimate()
    return {"value": round(linear_ops(w) / est / 1e12, 6), "unit": "TOPS", "cores": s.cores, "kind": "oracle",
            "sample": s.describe(), "pieces_timed": len(timed),
            "ms_per_piece": round(float(np.mean(timed)) * 1e3, 3), "est_step_s": round(est, 3), **s.breakdown()}


def run_reference(args, rank):
    """The oracle as it stands, on the host cores: W untimed pieces, then
    exactly K timed pieces, each one bounded piece of the workload (round robin
    over the selector of one image and the seven linears on a few rows).
    `steps` and `ms_per_step` describe those pieces as they ran; `value` is the
    throughput of the full step estimated from each piece's mean time
    (`est_step_s`, scaled to the whole workload)."""
    if rank != 0:
        return None
    w = wl.WORKLOADS[args.workload]
    s = OracleSampler(w, args.cpu_threads)
    n = len(s.pieces)
    for i in range(args.warmup):
        s.run_piece(i)
    warm = {i: list(v) for i, v in s.times.items()}
    s.times = {i: [] for i in range(n)}
    timed = []
    for i in range(args.steps):
        timed.append(s.run_piece(args.warmup + i))
    for i in range(n):  # a piece the timed round robin did not reach: its warm-up time, else one more run
        if not s.times[i]:
            s.times[i] = warm[i] or [s.run_piece(i)]
    est = s.estimate()
    value = linear_ops(w) / est / 1e12
    ms_piece = float(np.mean(timed)) * 1e3
    return {
        "metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_piece, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int4", "data": "synthetic", "impl": "reference",
        "config": {"workload": w.name, "B": w.B, "N": w.N, "d": w.d, "K": w.K, "T": w.T, "J": w.J, "M": w.M},
        "est_step_s": round(est, 3),
        "step_note": "each of the K steps is one piece of the workload (steps and ms_per_step describe the pieces "
                     "that ran); value = the full step's integer ops / est_step_s",
        "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": s.cores, "kind": "oracle",
                         "sample": "each step one piece: " + s.describe(), "est_step_s": round(est, 3),
                         **s.breakdown()},
        "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["p4q", "reference"], default="p4q")
    ap.add_argument("--workload", choices=sorted(wl.WORKLOADS), default=WORKLOAD.name,
                    help="workload of the step (default: the 32-image LLaVA-NeXT-13B batch)")
    ap.add_argument("--e2e-steps", type=int, default=50)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-threads", type=int, default=0, help="oracle threads (0 = all cores)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        rec = run_reference(args, rank)
    else:
        if world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group("nccl")
        rec = run_gpu(args, rank, world, local_rank)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
    if rec is not None:
        print(json.dumps(rec), flush=True)


if __name__ == "__main__":
    main()

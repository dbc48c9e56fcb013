"""The multi-process path of bench.py, on CPU with gloo at world size 2.

The hot path shards with no collective on the data path: every rank selects
and runs the linears on its own batch (its own input seed) with replicated
weights, and the only collective is the maximum over ranks of the timings,
from which rank 0 computes the whole-job throughput. The reference arm under
torchrun runs on rank 0 alone and prints one line.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2609_34867_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _max_worker(rank, world, port, outdir):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r took 10 + 5 r ms for its timed steps and 30 - 7 r ms end to end
        got = bench.max_over_ranks([10.0 + 5 * rank, 30.0 - 7 * rank], world, torch.device("cpu"))
        dist.barrier()
    finally:
        dist.destroy_process_group()
    with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
        json.dump(got, f)


def test_max_over_ranks_gloo_world_2(tmp_path):
    port = _free_port()
    mp.start_processes(_max_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    for r in range(2):
        assert json.load(open(tmp_path / f"rank{r}.json")) == [15.0, 30.0]


def test_max_over_ranks_single_process_is_identity():
    assert bench.max_over_ranks([1.5, 2.5], 1, torch.device("cpu")) == [1.5, 2.5]


def test_whole_job_throughput_counts_every_rank():
    w = wl.LLAVA15_7B
    ops = bench.linear_ops(w)
    one = bench.whole_job_tops(ops, 1, 0.5)
    assert np.isclose(one, ops / 0.5e-3 / 1e12)
    assert np.isclose(bench.whole_job_tops(ops, 4, 0.5), 4 * one)  # weak scaling: 4 batches in the same time


def test_ranks_draw_their_own_batches_and_share_weights():
    w = wl.Workload("t", B=2, N=64, d=128, K=8, T=4, J=3, seed=5, heavy_tail=False, linears=())
    s0, s1 = bench.rank_seed(w, 0), bench.rank_seed(w, 1)
    assert s0 == w.seed and s0 != s1
    x0, x1 = wl.selector_inputs(w, seed=s0), wl.selector_inputs(w, seed=s1)
    assert not np.array_equal(x0.V, x1.V) and not np.array_equal(x0.text, x1.text)
    # weights of a layer depend on the workload seed and layer only
    assert np.array_equal(wl.weight(128, 64, wl.weight_seed(w.seed, 0)), wl.weight(128, 64, wl.weight_seed(w.seed, 0)))


def test_reference_arm_under_torchrun_prints_once_from_rank_0():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "2", "--warmup", "3", "--workload", wl.LLAVA15_7B_ONE.name,
           "--cpu-threads", "2"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == 2
    assert rec["config"]["workload"] == wl.LLAVA15_7B_ONE.name
    assert rec["value"] > 0 and rec["cpu_baseline"]["kind"] == "oracle"
    assert rec["e2e"]["h2d_bytes_per_step"] == 0 and rec["e2e"]["d2h_bytes_per_step"] == 0

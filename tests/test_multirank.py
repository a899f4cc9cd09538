"""The multi-GPU host logic of bench.py on CPU: world_size 2 over gloo.

Weak scaling with no data-path collective: each rank draws its own sequences
(distinct seeds, same shapes), the job's time is the max over ranks (the only
collective), the whole-job rate counts every rank's bytes, and the reference
arm runs on rank 0 only.
"""
from __future__ import annotations

import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2607_05722_gb300 import workloads as W  # noqa: E402


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str) -> None:
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank's elapsed time differs; every rank must see the slowest
        ms = bench.max_over_ranks(1.5 + rank, world)
        dist.barrier()
        seed = bench.rank_seed(0, rank)
        wl = W.make_workload("tiny_b1_h4x1_d64_L256_bl8", seed=seed)
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{ms} {seed} {int(np.asarray(wl.attn.q_draft_bits).view(np.uint16).sum())}\n")
    finally:
        dist.destroy_process_group()


def test_two_ranks_reduce_max_and_draw_own_sequences(tmp_path):
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn")
    rows = [open(tmp_path / f"rank{r}.txt").read().split() for r in range(world)]
    ms = [float(r[0]) for r in rows]
    seeds = [int(r[1]) for r in rows]
    sums = [int(r[2]) for r in rows]
    assert ms == [2.5, 2.5], "every rank sees the slowest rank's time"
    assert seeds == [0, 1]
    assert sums[0] != sums[1], "ranks draw different sequences"


def test_single_rank_needs_no_collective():
    assert bench.max_over_ranks(3.25, 1) == 3.25


def test_job_rate_counts_every_rank():
    one = bench.job_kv_gbs(16_842_752, 2, 1, 0.0215)
    four = bench.job_kv_gbs(16_842_752, 2, 4, 0.0215)
    assert four == pytest.approx(4 * one)
    assert one == pytest.approx(2 * 16_842_752 / 21.5e-6 / 1e9)


def test_reference_arm_runs_on_rank_zero_only(capsys):
    class Args:
        steps, warmup, seed = 1, 0, 0
    assert bench.run_reference(Args(), 2, 1) is None
    assert capsys.readouterr().out == ""

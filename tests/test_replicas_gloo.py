"""The multi-GPU path is N independent replicas (one process per GPU, its own batch,
no exchange on the data path). Its host logic runs here on CPU as two gloo ranks: the
job's step time is the slowest rank's, throughput counts every rank's tokens, each rank
draws a different batch, and the reference arm runs on rank 0 only."""

import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2609_04010_gb300 import workloads as W
        ms = [0.5, 0.8][rank]                      # rank 1 is the slow replica
        ms_max = bench.max_over_ranks(ms, world)
        emitted = bench.sum_over_ranks(float(10 + rank), world)
        value = bench.whole_job_tokens_per_s(world, 8, 8, ms_max)
        ci = W.workload("tiny").accept_inputs(seed=rank)
        dist.barrier()
        out[rank] = (ms_max, emitted, value, int(ci.block_tokens.sum()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas():
    world = 2
    out = mp.Manager().dict()
    mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world,
                       start_method="spawn", join=True)
    (m0, e0, v0, t0), (m1, e1, v1, t1) = out[0], out[1]
    assert m0 == m1 == 0.8                         # the job waits for its slowest replica
    assert e0 == e1 == 21.0                        # emitted tokens add up over replicas
    assert v0 == v1 == pytest.approx(2 * 8 * 8 / 0.8e-3)
    assert t0 != t1                                # replicas verify different batches


def test_single_process_needs_no_group():
    import bench
    assert bench.max_over_ranks(1.25, 1) == 1.25
    assert bench.whole_job_tokens_per_s(1, 4, 2, 2.0) == pytest.approx(4000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    assert bench.main() == 0                       # returns at once: no oracle, no output

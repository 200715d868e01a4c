"""The rank logic of bench.py with two gloo ranks on CPU: max-over-ranks
timing, whole-job sums, and the reference arm printing on rank 0 only."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    mx = bench.max_over_ranks(float(10 + rank), world)
    sm = bench.sum_over_ranks(float(1 + rank), world)
    bench.barrier(world)

    class A:  # the reference arm returns at once on ranks other than 0
        workload = "tiny"
        warmup = 0
        steps = 1
    printed = bench.run_reference(A, rank, world) if rank != 0 else None
    out[rank] = (mx, sm, printed)
    dist.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    mp.start_processes(_worker, args=(2, _free_port(), out), nprocs=2, start_method="spawn")
    assert out[0][:2] == (11.0, 3.0)
    assert out[1] == (11.0, 3.0, None)

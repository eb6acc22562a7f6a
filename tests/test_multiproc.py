"""Host-side logic of the multi-GPU benchmark with two gloo ranks on CPU:
every rank runs its own batch (weak scaling, no collective on the data path),
the slowest rank's time is taken, and rank seeds give distinct batches."""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2606_05742_gb300 import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 100.0 + 7.0 * rank
        m = bench.max_over_ranks(local_ms)
        w = synth.make_workload(4, B=3, L=200, d=8, seed=bench.rank_seed(0, rank))
        out[rank] = (m, bench.job_throughput(world, 50, m), int(w.tokens.sum()))
    finally:
        dist.destroy_process_group()


def test_two_ranks_max_time_and_throughput():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    assert out[0][0] == out[1][0] == 107.0          # slowest rank
    assert out[0][1] == pytest.approx(2 * 50 / 0.107)
    assert out[0][2] != out[1][2]                    # each rank its own batch


def test_single_process_passthrough():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(1, 10, 20.0) == pytest.approx(500.0)

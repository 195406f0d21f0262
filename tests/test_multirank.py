"""World-size-2 checks (gloo, CPU) of the benchmark's multi-rank bookkeeping: every rank its own
document, max-over-ranks timing, whole-job throughput. No data-path collective exists."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 100.0 + 50.0 * rank          # rank 1 is the slowest
        m = bench.max_over_ranks(ms, dist, "cpu")
        out[rank] = (m, bench.doc_seed(rank), bench.throughput(world, 8192, 5, m))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_timing_and_sharding():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    assert out[0][0] == out[1][0] == 150.0
    assert out[0][1] != out[1][1]                      # distinct documents per rank
    assert out[0][2] == pytest.approx(2 * 8192 * 5 / 0.150)


def test_single_rank_passthrough():
    assert bench.max_over_ranks(3.5, None, "cpu") == 3.5
    assert bench.throughput(1, 100, 2, 1000.0) == pytest.approx(200.0)

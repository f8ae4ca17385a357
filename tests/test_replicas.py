"""The multi-GPU path is replicas only (every rank runs its own P learners, no
data-path collective): the host logic that joins the ranks' timings, run as two
gloo processes on CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, ws, port, seconds, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method="env://", rank=rank, world_size=ws)
    try:
        assert bench.dist_env() == (ws, rank, rank)
        dist.barrier()
        t = bench.job_seconds(seconds[rank], ws)
        out[rank] = (t, bench.replica_throughput(ws, 8192, 5, t))
    finally:
        dist.destroy_process_group()


def test_job_time_is_the_slowest_rank():
    ws, port = 2, _free_port()
    seconds = [0.75, 1.25]
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(ws, port, seconds, out), nprocs=ws, join=True)
    for rank in range(ws):
        t, value = out[rank]
        assert t == max(seconds)
        assert value == pytest.approx(ws * 8192 * 5 / max(seconds))


def test_single_rank_needs_no_process_group():
    assert bench.job_seconds(0.5, 1) == 0.5
    assert bench.replica_throughput(1, 100, 4, 2.0) == 200.0

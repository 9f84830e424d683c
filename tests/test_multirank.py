"""Host logic of the N > 1 bench path on CPU ranks (gloo, world size 2).

The operator shards over (b, h) with no exchange, so an N-GPU run is N
replicas: each rank times its own replica, the ranks agree on the slowest
time (max-reduce), and the job value counts the work of every rank.  These
tests run that reduction over a real two-process gloo group.
"""
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


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 2.0 + 3.0 * rank  # rank 1 is the slow one
        slowest = bench.reduce_max(ms, world, torch.device("cpu"))
        out[rank] = (slowest, bench.job_value(1e12, world, slowest))
    finally:
        dist.destroy_process_group()


def test_two_rank_max_reduce_and_job_value():
    world, port = 2, _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, join=True, start_method="spawn")
    assert out[0][0] == out[1][0] == 5.0
    # 2 replicas x 1e12 flops each over 5 ms = 400 TFLOP/s, the same on every rank
    assert out[0][1] == out[1][1] == pytest.approx(400.0)


def test_single_rank_is_local_time():
    assert bench.reduce_max(1.25, 1, torch.device("cpu")) == 1.25
    assert bench.job_value(6e12, 1, 10.0) == pytest.approx(600.0)

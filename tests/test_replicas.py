"""The multi-GPU form of the benchmark is independent replicas: the job time is
the slowest rank's and the throughput counts every rank's payload.  Checked
with two gloo ranks on CPU."""
import os
import socket

import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, out):
    import torch.distributed as dist

    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, value = bench.replica_timing(100.0 + 50.0 * rank, 10**9, 10, world, "cpu")
        out[rank] = (ms, value)
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas_take_the_max_time_and_sum_the_payload():
    world = 2
    mgr = mp.get_context("spawn").Manager()  # no fork of a process that may hold threads
    out = mgr.dict()
    mp.spawn(_rank, args=(world, _free_port(), out), nprocs=world, join=True)
    for r in range(world):
        ms, value = out[r]
        assert ms == 150.0                       # the slower rank's time
        assert abs(value - 2 * 1e9 / 0.015 / 1e9) < 1e-6  # both ranks' bytes / that time


def test_single_process_needs_no_group():
    import bench
    ms, value = bench.replica_timing(20.0, 10**9, 4, 1)
    assert ms == 20.0 and abs(value - 1e9 / 0.005 / 1e9) < 1e-9

"""Multi-GPU in this path is "replicas only" (independent sequences on independent GPUs, no
collective on the data path). The bench's cross-rank aggregation -- every rank's tokens over the
slowest rank's timed region -- is checked here with two gloo ranks on the CPU."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    local_ms = [100.0, 250.0][rank]
    local_tokens = [512, 512][rank]
    max_ms, total, value = bench.aggregate_ranks(local_ms, local_tokens, dist, "cpu")
    out[rank] = (max_ms, total, value)
    dist.barrier()
    dist.destroy_process_group()


def test_replica_throughput_is_total_tokens_over_slowest_rank():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()  # no fork of this (threaded) test process
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        max_ms, total, value = out[r]
        assert max_ms == 250.0 and total == 1024
        assert abs(value - 1024 / 0.25) < 1e-9


def test_single_process_aggregation_is_local():
    import bench

    assert bench.aggregate_ranks(200.0, 512) == (200.0, 512, 2560.0)

"""The multi-rank (replica) logic of bench.py on CPU: two gloo ranks (world size 2)
reduce their timed-region durations to the slowest one and report the whole job's
tokens over that time.  No GPU: each rank only times a host-side wait."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 100.0 + 50.0 * rank          # rank 1 is the slow one
    slow = bench.slowest_rank_ms(ms, world, device="cpu")
    value = bench.job_tokens_per_s(world, 8192, 5, slow)
    dist.barrier()
    out[rank] = (slow, value)
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1]
    slow, value = res[0]
    assert slow == 150.0
    assert value == pytest.approx(2 * 8192 * 5 / 0.150)


def test_single_rank_is_identity():
    import bench
    assert bench.slowest_rank_ms(12.5, 1) == 12.5
    assert bench.job_tokens_per_s(1, 1000, 2, 500.0) == pytest.approx(4000.0)

"""The multi-GPU form of the server-hierarchical strategy (one replica per rank, period-end
averaging as an all-reduce mean), run with two gloo ranks on CPU tensors."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2406_14898_gb300.hierarchical import allreduce_mean_
    g = torch.Generator().manual_seed(100 + rank)
    w = torch.randn(1000, generator=g, dtype=torch.float32)
    mine = w.clone()
    allreduce_mean_(w)
    out[rank] = (mine.numpy(), w.numpy())
    dist.destroy_process_group()


def test_allreduce_mean_of_two_replicas():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    mean = (res[0][0] + res[1][0]) / 2
    np.testing.assert_allclose(res[0][1], mean, rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(res[0][1], res[1][1])

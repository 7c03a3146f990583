"""The multi-GPU form of the server-hierarchical strategy (one replica per rank, period-end
averaging as an all-reduce followed by the library's 1/ranks scaling), run with two gloo
ranks on CPU tensors.  The server is a host-side stand-in that records the calls and
applies the scaling the library's fl_server_average_finish applies (fp32 multiply by
1/n), so the call order and the rank count handed to the library are what is tested."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


class _FakeServer:
    def __init__(self, w):
        self.w = w
        self.calls = []

    def sync(self):
        self.calls.append("sync")

    def average_finish(self, n):
        import torch
        self.calls.append(("finish", n))
        self.w.mul_(torch.tensor(1.0 / n, dtype=torch.float32))


def _rank(rank, world, port, out):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2406_14898_gb300.hierarchical import average_across_ranks
    g = torch.Generator().manual_seed(100 + rank)
    w = torch.randn(1000, generator=g, dtype=torch.float32)
    mine = w.clone()
    srv = _FakeServer(w)
    average_across_ranks(srv, arena=w)
    out[rank] = (mine.numpy(), w.numpy(), srv.calls)
    dist.destroy_process_group()


def test_average_across_two_ranks():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    mean = (res[0][0] + res[1][0]) * np.float32(0.5)
    np.testing.assert_array_equal(res[0][1], mean)
    np.testing.assert_array_equal(res[0][1], res[1][1])
    for r in range(world):
        assert res[r][2] == ["sync", ("finish", world), "sync"]

"""The multi-GPU form of the server-hierarchical strategy (replicas on every rank, period-end
averaging as the in-handle mean, an all-reduce, then the library's 1/ranks scaling), run
with two gloo ranks of two replicas each on CPU tensors.  The server is a host-side
stand-in that records the calls and applies the arithmetic of the library's
fl_server_average_replicas (fp32 sum in replica order times 1/n) and
fl_server_average_finish (fp32 multiply by 1/n), so the call order and the counts handed
to the library are what is tested."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


class _FakeServer:
    """Holds n_rep replicas' weights back to back in w, as a handle with cfg.n_replicas."""

    def __init__(self, w, n_rep):
        self.w = w
        self.n_rep = n_rep
        self.calls = []

    def sync(self):
        self.calls.append("sync")

    def average_replicas(self):
        import torch
        self.calls.append("replicas")
        v = self.w.view(self.n_rep, -1)
        s = v[0].clone()
        for r in range(1, self.n_rep):
            s += v[r]
        v.copy_((s * torch.tensor(1.0 / self.n_rep, dtype=torch.float32)).expand_as(v))

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
    w = torch.randn(2 * 500, generator=g, dtype=torch.float32)  # two replicas on each rank
    mine = w.clone()
    srv = _FakeServer(w, 2)
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
    half = np.float32(0.5)
    rank_means = [(res[r][0][:500] + res[r][0][500:]) * half for r in range(world)]
    mean = (rank_means[0] + rank_means[1]) * half
    for r in range(world):
        np.testing.assert_array_equal(res[r][1][:500], mean)
        np.testing.assert_array_equal(res[r][1][500:], mean)
        assert res[r][2] == ["replicas", "sync", ("finish", world), "sync"]

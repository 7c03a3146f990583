"""Server-hierarchical training (§3.3 of the paper): one server replica per client, the
replicas trained side by side and their parameters averaged at the end of every period.

On one GPU the replicas are independent fl_server handles, each on its own CUDA stream, so
their kernels can overlap; fl_server_average forms the mean on the device.  Across GPUs
(one replica per rank) the mean is an all-reduce (sum) of each replica's fp32 master-weight
arena, then fl_server_average_finish scales it by 1/ranks and refreshes the bf16 working
copy.  All arithmetic runs in the CUDA library or in the collective; this module only
orders the calls.
"""
from __future__ import annotations

from typing import List, Sequence

from . import flglm as F


class _ArenaView:
    """__cuda_array_interface__ of a library-owned fp32 device array (no copy)."""

    def __init__(self, ptr: int, n: int):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": "<f4", "data": (ptr, False), "version": 2,
                                         "strides": None}


def arena_tensor(server: F.Server):
    """A torch tensor aliasing the server's fp32 master weights (valid while the server lives)."""
    import torch
    ptr, n = server.param_arena()
    return torch.as_tensor(_ArenaView(ptr, n), device="cuda")


def allreduce_sum_(tensor, group=None):
    """In-place sum of `tensor` over the ranks of `group` (the collective alone)."""
    import torch.distributed as dist
    dist.all_reduce(tensor, op=dist.ReduceOp.SUM, group=group)
    return tensor


def average_across_ranks(server, group=None, arena=None):
    """Period-end averaging with one replica per rank: all-reduce (sum) of the master
    weights, then the library scales the sum by 1/ranks and refreshes the bf16 working copy.
    `arena` (default: the server's master arena as a CUDA tensor) is the buffer the
    collective sums."""
    import torch
    import torch.distributed as dist
    server.sync()
    w = arena_tensor(server) if arena is None else arena
    allreduce_sum_(w, group)
    if w.is_cuda:
        torch.cuda.synchronize()
    server.average_finish(dist.get_world_size(group))
    server.sync()


class HierarchicalServers:
    """K replicas of the server on one GPU, replica k serving client k."""

    def __init__(self, cfg: F.fl_server_cfg, seed: int, n_replicas: int):
        import torch
        self.streams = [torch.cuda.Stream() for _ in range(n_replicas)]
        # same seed: every replica starts from the same parameters, as after an averaging
        self.replicas: List[F.Server] = [F.Server(cfg, seed, stream=s) for s in self.streams]

    def step(self, client_states: Sequence, seq_lens: Sequence[int], out_states: Sequence, grad_out: Sequence,
             grad_in: Sequence, lr: float):
        """One training step of every replica on its own client (forward, backward and
        AdamW), each on its own stream."""
        for k, srv in enumerate(self.replicas):
            srv.forward([client_states[k]], [seq_lens[k]], [out_states[k]])
        for k, srv in enumerate(self.replicas):
            srv.backward_step([grad_out[k]], [grad_in[k]], lr)

    def average(self):
        F.fl_server_average(self.replicas)

    def sync(self):
        for srv in self.replicas:
            srv.sync()

    def close(self):
        for srv in self.replicas:
            srv.close()
        self.replicas = []

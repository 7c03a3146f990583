"""Server-hierarchical training (§3.3 of the paper): one server replica per client, the
replicas trained side by side and their parameters averaged at the end of every period.

On one GPU the replicas are either independent fl_server handles, each on its own CUDA
stream, averaged by fl_server_average (HierarchicalServers), or up to four replicas held in
one handle (cfg.n_replicas), whose block GEMMs run as one batched launch per GEMM and which
fl_server_average_replicas averages (BatchedReplicas; every replica's clients must hold the
same number of tokens).  Across GPUs (replicas on every rank) the mean is the in-handle
mean, then an all-reduce (sum) of each rank's fp32 master-weight arena, then
fl_server_average_finish scales it by 1/ranks and refreshes the bf16 working copy (with an
equal number of replicas on every rank, the mean of the ranks' means is the mean over all
replicas).  All arithmetic runs in the CUDA library or in the collective; this module only
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
    """Period-end averaging with the replicas of `server` on every rank: the replicas held in
    the handle are averaged first (nothing to do with one), then the master weights are
    all-reduced (sum) and the library scales the sum by 1/ranks and refreshes the bf16
    working copy.  `arena` (default: the server's master arena as a CUDA tensor) is the
    buffer the collective sums."""
    import torch
    import torch.distributed as dist
    server.average_replicas()
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


class BatchedReplicas:
    """n_replicas (2..4) server replicas in one handle: a call's K clients are split in
    order into n_replicas groups holding the same number of tokens, group r trained by
    replica r; every block GEMM of all replicas is one batched launch."""

    def __init__(self, cfg: F.fl_server_cfg, seed: int, n_replicas: int, stream=None):
        c = F.fl_server_cfg.from_buffer_copy(cfg)
        c.n_replicas = n_replicas
        self.n_replicas = n_replicas
        # every replica starts from the same parameters, as after an averaging
        self.server = F.Server(c, seed, stream=stream)

    def step(self, client_states: Sequence, seq_lens: Sequence[int], out_states: Sequence, grad_out: Sequence,
             grad_in: Sequence, lr: float):
        """One training step of every replica on its group of clients."""
        self.server.forward(client_states, seq_lens, out_states)
        self.server.backward_step(grad_out, grad_in, lr)

    def average(self):
        self.server.average_replicas()

    def get_param(self, replica: int, block: int, tensor_id: int):
        return self.server.get_replica_param(replica, block, tensor_id)

    def sync(self):
        self.server.sync()

    def close(self):
        self.server.close()

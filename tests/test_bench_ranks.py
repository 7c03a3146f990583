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


def test_stored_traffic_used_only_for_the_current_gemm_sources(tmp_path):
    """The roofline's DRAM traffic comes from a committed ncu summary only while the GEMM
    sources it was measured on are unchanged (their fingerprint is in the summary) and
    only for the workload it names."""
    import bench
    fp = bench.kernel_version()
    good = tmp_path / "gemm_x_stack26.md"
    good.write_text(f"fingerprint: {fp}\ntraffic_bytes_per_launch: 123456\n")
    assert bench.ncu_traffic(str(good), "stack26")["bytes_per_launch"] == 123456
    assert bench.ncu_traffic(str(good), "block6b") is None            # another workload
    stale = tmp_path / "gemm_y_stack26.md"
    stale.write_text("fingerprint: 0000000000000000\ntraffic_bytes_per_launch: 123456\n")
    assert bench.ncu_traffic(str(stale), "stack26") is None            # other GEMM sources
    assert bench.ncu_traffic(str(tmp_path / "missing_stack26.md"), "stack26") is None

"""The multi-GPU benchmark path runs one independent replica per rank: no
data-path collective, only the harness's barrier and the max-over-ranks time.
Two gloo ranks on the CPU check that aggregation: every rank sees the slowest
rank's time, and the whole-job value counts both ranks' bytes."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        dist.barrier()
        total_ms = 100.0 if rank == 0 else 250.0  # rank 1 is the slow replica
        ms_step, value = bench.aggregate(total_ms, 10, 1_000_000_000, world, torch.device("cpu"))
        results[rank] = (ms_step, value)
    finally:
        dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    results = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, results)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(2):
        ms_step, value = results[r]
        assert ms_step == pytest.approx(25.0)
        assert value == pytest.approx(2 * 1.0 / 0.025)  # 2 ranks x 1 GB per 25 ms


def test_single_rank_needs_no_process_group():
    import bench
    ms_step, value = bench.aggregate(50.0, 5, 2_000_000_000, 1, torch.device("cpu"))
    assert ms_step == 10.0 and value == pytest.approx(200.0)

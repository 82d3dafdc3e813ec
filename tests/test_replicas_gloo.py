"""The multi-GPU form of the benchmark is N independent replicas (the convolution path has
no exchange step): the only cross-rank steps are a barrier and the max of the timed
duration. This runs that host logic with 2 gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local_ms = 100.0 + 50.0 * rank          # rank 1 is the slow replica
    dist.barrier()
    worst = bench.max_over_ranks(local_ms, "cpu")
    tops = bench.job_tops(2e12, 10, world, worst)
    q.put((rank, worst, tops))
    dist.destroy_process_group()


def test_two_replicas_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, worst, tops in out:
        assert worst == pytest.approx(150.0)
        # 2 ranks x 2e12 ops x 10 steps in 150 ms
        assert tops == pytest.approx(2 * 2e12 * 10 / 0.150 / 1e12)


def test_single_process_needs_no_collective():
    import bench
    assert bench.max_over_ranks(3.5, "cpu") == 3.5
    assert bench.job_tops(1e12, 4, 1, 2.0) == pytest.approx(2000.0)

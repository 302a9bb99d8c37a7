"""Multi-rank host logic of bench.py on CPU: two gloo ranks (the data path has no collective; the
ranks are independent replicas), whose timed regions differ, agree on the job's time (the slowest
rank's) and on the whole-job throughput (units of all ranks over that time)."""
import os
import socket

import pytest
import torch.multiprocessing as tmp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, local_ms, q):
    import torch.distributed as dist

    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.slowest_rank_ms(local_ms[rank], dist)
        q.put((rank, ms, bench.job_throughput(50, world, ms)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_slowest_time_and_job_throughput():
    world = 2
    local_ms = [120.0, 150.0]
    ctx = tmp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, local_ms, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [150.0, 150.0]
    assert all(r[2] == pytest.approx(50 * 2 / 0.150) for r in res)


def test_single_rank_is_its_own_job():
    import bench
    assert bench.slowest_rank_ms(42.0, None) == 42.0
    assert bench.job_throughput(10, 1, 20.0) == pytest.approx(500.0)

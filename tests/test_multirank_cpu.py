"""The multi-rank bench logic on CPU: two gloo ranks, each timing its own shard.

The encode/decode units (l, s, b, h) are independent, so ranks exchange no data; the job
value is the sum of the ranks' bytes over the slowest rank's time.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ws, r, local = bench._dist()
        ms = [3.0, 5.0][rank]  # rank 1 is the slower one
        slowest = bench.rank_reduce(ms, "max")
        fastest = bench.rank_reduce(ms, "min")
        value = bench.job_throughput(1_000_000_000, ws, slowest)
        q.put((rank, ws, r, local, slowest, fastest, value))
    finally:
        dist.destroy_process_group()


def test_two_ranks_max_time_and_job_value():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(q.get(timeout=5) for _ in range(2))
    for rank, ws, r, local, slowest, fastest, value in res:
        assert (ws, r, local) == (2, rank, rank)
        assert slowest == 5.0 and fastest == 3.0
        # 2 ranks x 1 GB in 5 ms
        assert value == pytest.approx(400.0)


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.rank_reduce(7.5, "max") == 7.5
    assert bench.job_throughput(2_000_000_000, 1, 1.0) == pytest.approx(2000.0)

"""Host logic of bench.py's multi-GPU path (replicas only), run as two gloo
ranks on the CPU: every rank times its own replica; the reported times are
the maximum over ranks and the throughput counts every rank's tokens."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import sys
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    times = [10.0 + 5.0 * rank, 2.0 + rank]  # rank 1 is the slower one
    value, out = bench.aggregate(times, 32768, world)
    q.put((rank, value, out))
    dist.destroy_process_group()


def test_aggregate_takes_max_over_ranks_and_sums_tokens():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, value, out in res:
        assert out == [15.0, 3.0]
        assert value == pytest.approx(2 * 32768 / 15e-3)


def test_single_rank_aggregate():
    import bench
    value, out = bench.aggregate([4.0], 1000, 1)
    assert out == [4.0] and value == pytest.approx(1000 / 4e-3)

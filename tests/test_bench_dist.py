"""The N>1 bench aggregation on CPU: two gloo ranks, each a replica of the
workload (weak scaling), job time = slowest rank, value = sum over ranks."""
import os
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rank(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    secs = [2.0, 3.0][rank]
    slow = bench.reduce_max(secs, dist, "cpu")
    val = bench.job_throughput(10 ** 9, 4, world, slow)
    dist.barrier()
    q.put((rank, slow, val))
    dist.destroy_process_group()


def test_two_rank_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29517
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [3.0, 3.0]
    # 2 ranks x 4 steps x 1 GB over the slowest rank's 3 s
    assert res[0][2] == pytest.approx(8.0 / 3.0)


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(1.5) == 1.5
    assert bench.job_throughput(2 * 10 ** 9, 5, 1, 2.0) == pytest.approx(5.0)

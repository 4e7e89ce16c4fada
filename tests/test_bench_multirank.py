"""The N > 1 path of bench.py without a GPU: two gloo ranks on the CPU.

bench.py runs one independent replica of the workload per rank (token batches are independent,
Algorithm 2 acts on each token separately), so its only cross-rank step is the aggregation: the
job time is the slowest rank's time and the job throughput sums the ranks' tokens over it.
"""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, ms, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench._DIST = dist
        slowest = bench._max_over_ranks(ms[rank])
        q.put((rank, slowest, bench._job_value(world, 8, 1000, slowest)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_sum_the_tokens():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ms = [3.0, 5.0]          # rank 1 is slower
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, ms, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    for p in procs:
        if p.is_alive():
            p.kill()
    assert all(p.exitcode == 0 for p in procs)
    got = dict((r, (t, v)) for r, t, v in (q.get(timeout=10) for _ in range(2)))
    for r in range(2):
        assert got[r][0] == pytest.approx(5.0)                    # every rank sees the max
        assert got[r][1] == pytest.approx(2 * 8 * 1000 / 5e-3)    # both ranks' tokens / slowest time


def test_single_process_aggregation_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    bench._DIST = None
    assert bench._max_over_ranks(4.25) == 4.25
    assert bench._job_value(1, 8, 100, 2.0) == pytest.approx(8 * 100 / 2e-3)

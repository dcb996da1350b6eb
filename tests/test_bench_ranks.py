"""The bench's multi-rank path on CPU (gloo, world size 2): the timed region
is the slowest rank's, `value` counts every rank's units over it, and the
reference arm runs on rank 0 only (the path shards into independent
replicas; there is no collective on the data path)."""
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
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, rate = bench.job_rate(10.0 * (rank + 1), 1e9, world, "cpu")
        q.put((rank, ms, rate))
    finally:
        dist.destroy_process_group()


def test_job_rate_takes_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for _, ms, rate in got:
        assert ms == pytest.approx(20.0)
        assert rate == pytest.approx(2 * 1e9 / 0.020)


def test_single_rank_rate():
    sys.path.insert(0, ROOT)
    import bench
    ms, rate = bench.job_rate(4.0, 8e6, 1, "cpu")
    assert ms == 4.0 and rate == pytest.approx(2e9)


def test_reference_arm_only_on_rank0():
    sys.path.insert(0, ROOT)
    import bench

    class A:
        steps, warmup = 1, 0
    assert bench.run_reference(A(), 1, 2) is None

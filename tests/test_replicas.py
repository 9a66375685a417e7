"""Replicas across ranks (CPU, gloo, world_size 2): bench.py's whole-job
numbers take the max of the ranks' timed totals and count every rank's images.
Images are independent, so the data path has no collective; this is the only
cross-rank step."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        total_ms = [10.0, 12.5][rank]
        e2e_ms = [30.0, 20.0][rank]
        out = bench.combine_ranks(total_ms, e2e_ms, images_per_rank=4, world=world,
                                  device=torch.device("cpu"))
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


def test_combine_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank in (0, 1):
        total, e2e, rate, e2e_rate = res[rank]
        assert total == pytest.approx(12.5) and e2e == pytest.approx(30.0)
        assert rate == pytest.approx(8 / 12.5e-3)        # 2 ranks x 4 images over the slowest
        assert e2e_rate == pytest.approx(8 / 30.0e-3)


def test_combine_ranks_single():
    import bench
    total, e2e, rate, e2e_rate = bench.combine_ranks(5.0, 8.0, 3, 1, torch.device("cpu"))
    assert (total, e2e) == (5.0, 8.0) and rate == pytest.approx(600.0)

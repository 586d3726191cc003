"""Host-side logic of the multi-GPU bench on CPU: two gloo ranks.

Each rank gets its own sequences (sharded seeds, no data-path collective) and
the reported time is the slowest rank's, identical on every rank.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(10.0 + 5.0 * rank, dist, torch.device("cpu"))
        q.put((rank, ms, bench.shard_seeds(rank), bench.job_rows_per_s(world, 512, 4, ms)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_inputs_and_take_max_time(repo_root):
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, s0, v0), (r1, ms1, s1, v1) = res
    assert ms0 == ms1 == 15.0                       # the slowest rank's time, on every rank
    assert not set(s0) & set(s1)                    # disjoint input shards
    assert v0 == v1 == pytest.approx(2 * 512 * 4 / 15e-3)


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, None, None) == 3.5
    assert bench.job_rows_per_s(1, 512, 10, 1.0) == pytest.approx(512 * 10 / 1e-3)

"""Host logic of the N > 1 path (independent replicas, weak scaling) on CPU
with two gloo ranks: the barrier, the max over ranks of the timed region and
the whole-job throughput.  No GPU and no data-path collective is involved:
each replica serves its own sequences."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        t_local = 1.0 + 0.5 * rank          # rank 1 is the slower replica
        t_max = bench.max_over_ranks(t_local, world)
        value = bench.aggregate_tokens_per_s(3.0, 100, t_max, world)
        bench.barrier(world)
        out.put((rank, t_max, value))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_replica():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, t_max, value in res:
        assert t_max == pytest.approx(1.5)
        # 2 replicas x 3 tokens per step x 100 steps in 1.5 s
        assert value == pytest.approx(2 * 3.0 * 100 / 1.5)


def test_single_rank_needs_no_process_group():
    import bench

    assert bench.max_over_ranks(2.5, 1) == 2.5
    assert bench.aggregate_tokens_per_s(2.0, 10, 4.0, 1) == pytest.approx(5.0)

"""The multi-GPU mode of bench.py is N independent replicas (the path has no exchange
step): a barrier around the timed region and the maximum of the ranks' times.  This runs
that reduction with two gloo ranks on the CPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as tmp

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist

    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        dist.barrier()
        out[rank] = (bench._max_over_ranks(10.0 + 5.0 * rank, world),
                     bench.replica_value(1000.0, world, bench._max_over_ranks(10.0 + 5.0 * rank, world)),
                     # the end-to-end leg's go / no-go: one rank short of host memory stops both
                     bench._max_over_ranks(1.0 if rank == 1 else 0.0, world))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas_agree_on_the_slowest_time():
    ctx = tmp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0           # max over the ranks' times
    assert res[0][1] == pytest.approx(2 * 1000.0 / 0.015)   # N x units / slowest time
    assert res[0][2] == res[1][2] == 1.0            # both ranks skip the end-to-end leg together


def test_single_rank_is_the_identity():
    import bench

    assert bench._max_over_ranks(3.5, 1) == 3.5
    assert bench.replica_value(100.0, 1, 50.0) == pytest.approx(2000.0)

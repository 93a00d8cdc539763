"""The benchmark's multi-rank logic on CPU ranks (gloo, world size 2).

The AdamW step has no cross-rank exchange: with N ranks every rank runs its
own replica of the workload (weak scaling), the timed region is bracketed by
barriers, the job's time is the slowest rank's, and the reported throughput
is the units all ranks processed over that time. Here two gloo ranks report
different times; both must see the maximum, and rank 0's whole-job value
must count both replicas.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        ms = [3.0, 5.5][rank]
        dist.barrier()
        got = bench.max_over_ranks(ms)
        out[rank] = (got, bench.job_value(1_000_000, world, got))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    import torch.multiprocessing as mp
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    old = os.environ.get("PYTHONPATH", "")
    os.environ["PYTHONPATH"] = root + (os.pathsep + old if old else "")
    try:
        ctx = mp.get_context("spawn")
        out = ctx.Manager().dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
        assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    finally:
        os.environ["PYTHONPATH"] = old
    for r in range(2):
        ms, value = out[r]
        assert ms == 5.5
        assert value == pytest.approx(2 * 1_000_000 / 5.5e-3)


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(4.25) == 4.25
    assert bench.job_value(10, 1, 2.0) == pytest.approx(5000.0)

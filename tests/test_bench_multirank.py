"""The multi-rank aggregation of bench.py on CPU (gloo, world size 2): the
job's throughput is every rank's tokens over the slowest rank's time."""
import os

import pytest
import torch.multiprocessing as mp


def _worker(rank, world, port, q):
    import torch
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 10.0 if rank == 0 else 20.0        # rank 1 is the slow one
    e2e = 0.5 if rank == 0 else 0.25
    value, e2e_value, t_max = bench.aggregate_ranks(1.0e9, ms, 2.0e8, e2e, world, device="cpu")
    q.put((rank, value, e2e_value, t_max))
    torch.distributed.destroy_process_group()


def test_aggregate_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + os.getpid() % 1000
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for _, value, e2e_value, t_max in res:
        assert t_max == 20.0
        assert value == pytest.approx(2 * 1.0e9 / 0.020)
        assert e2e_value == pytest.approx(2 * 2.0e8 / 0.5)


def test_single_rank_needs_no_process_group():
    import bench
    value, e2e_value, t_max = bench.aggregate_ranks(3.0e9, 30.0, 1.0e8, 0.1, 1)
    assert (value, e2e_value, t_max) == (pytest.approx(1.0e11), pytest.approx(1.0e9), 30.0)

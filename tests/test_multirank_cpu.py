"""The benchmark's multi-rank path on CPU: two gloo ranks, weak-scaling replicas.

Each rank times its own replica; the job time is the maximum over ranks and
the reported throughput is the units of all ranks divided by it.  No GPU and
no collective on the data path are involved.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, out):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local = [10.0 + 5.0 * rank, 3.0 - rank]          # per-rank (total ms, kernel ms)
        out[rank] = (bench.reduce_max_over_ranks(local), bench.replica_seed(100, rank))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_max_and_distinct_seeds():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    (m0, s0), (m1, s1) = out[0], out[1]
    assert m0 == m1 == [15.0, 3.0]
    assert s0 != s1
    # whole-job throughput: both ranks' units over the slowest rank's time
    units_per_rank = 7.0e9
    assert 2 * units_per_rank / (m0[0] / 1e3) == pytest.approx(2 * 7.0e9 / 0.015)


def test_single_process_is_identity():
    import bench
    assert bench.reduce_max_over_ranks([1.5, 2.5]) == [1.5, 2.5]

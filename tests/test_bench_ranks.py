"""bench.py's whole-job numbers over N replicas (one rank per GPU): every rank
takes the slowest rank's time (max over ranks) and the value counts the units
all ranks processed.  Run here as two gloo ranks on the CPU."""
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
        ms_local = [40.0, 50.0][rank]
        out[rank] = bench.job_rate(ms_local, world, flops_per_rank_step=2e12, steps=10,
                                   device="cpu")
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_all_work():
    ctx = mp.get_context("spawn")
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
    for r in range(2):
        value, ms_max = res[r]
        assert ms_max == 50.0
        # 2 ranks x 10 steps x 2e12 flop in 50 ms
        assert value == pytest.approx(2 * 10 * 2e12 / 0.050 / 1e12)


def test_one_rank_needs_no_process_group():
    import bench
    value, ms_max = bench.job_rate(25.0, 1, 1e12, 4, device="cpu")
    assert ms_max == 25.0 and value == pytest.approx(4 * 1e12 / 0.025 / 1e12)

"""The N > 1 path of bench.py on the CPU: replicas with no data-path
collective; the job's time is the slowest rank's and its counts the sum over
ranks (world size 2, gloo, 127.0.0.1)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, counts = bench.job_totals(10.0 + 5.0 * rank, (3 + rank, 100 * (rank + 1)), world, "cpu")
        ms_e, empty = bench.job_totals(7.0 * (rank + 1), (), world, "cpu")
        out[rank] = (ms, counts, ms_e, empty, bench.job_value(32, world, 20, ms))
    finally:
        dist.destroy_process_group()


def test_job_totals_over_two_gloo_ranks():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    for r in (0, 1):
        ms, counts, ms_e, empty, value = res[r]
        assert ms == 15.0                      # the slower rank's time
        assert counts == [7, 300]              # summed over ranks
        assert ms_e == 14.0 and empty == []
        assert value == pytest.approx(32 * 2 * 20 / 0.015)


def test_single_rank_is_unchanged():
    import bench
    assert bench.job_totals(4.0, (1, 2), 1, "cpu") == (4.0, [1, 2])
    assert bench.job_value(32, 1, 20, 10.0) == pytest.approx(64000.0)

"""The N > 1 path of bench.py on the CPU: two ranks over gloo.

Units are independent, so ranks shard them with no collective on the data
path; the only exchange is the max over ranks of the measured times.  These
tests run the bench's own rank helpers in two spawned processes.
"""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as tmp

import bench
import grkv_inputs as gi


def _free_port() -> int:
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = bench.rank_workload(gi.workload(1).replace(units=2, n=64, budget=40), rank, world)
        q, k, v = gi.unit_arrays(wl, 0)
        # a rank-dependent "measured" time: the job's time is the slowest rank's
        ms, e2e = bench.max_over_ranks([1.0 + rank, 10.0 - rank], dist)
        out[rank] = {"seed": wl.seed, "k00": float(np.asarray(k, dtype=np.float64)[0, 0]),
                     "ms": ms, "e2e": e2e,
                     "value": bench.job_throughput(wl.units, wl.n, world, ms)}
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_ranks_shard_units_and_take_the_max_time():
    world = 2
    with tmp.Manager() as mgr:
        out = mgr.dict()
        tmp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert set(res) == {0, 1}
    # independent units per rank: different seeds and different data
    assert res[0]["seed"] != res[1]["seed"]
    assert res[0]["k00"] != res[1]["k00"]
    # every rank sees the slowest rank's time, element-wise
    for r in (0, 1):
        assert res[r]["ms"] == 2.0 and res[r]["e2e"] == 10.0
    # whole-job throughput counts both ranks' units over the max time
    assert res[0]["value"] == pytest.approx(2 * 64 * 2 / 2e-3)


def test_single_rank_helpers_are_identities():
    wl = gi.workload(1)
    assert bench.rank_workload(wl, 0, 1) is wl
    assert bench.max_over_ranks([3.0, 4.5]) == [3.0, 4.5]
    assert bench.job_throughput(256, 32768, 1, 1.0) == pytest.approx(256 * 32768 / 1e-3)

"""Multi-process host logic of bench.py on CPU (gloo, world size 2).

Each rank prunes its own shard of samples with no collective on the data path;
only the timing bookkeeping (barrier, max over ranks, sum of units) crosses
ranks. This checks that bookkeeping without a GPU.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    d = bench.Dist()
    d.init("gloo")
    d.barrier()
    sec = 1.0 + rank            # rank 1 is the slow one
    units = 8.0 * (rank + 1)    # and processed more samples
    mx = d.max(sec)
    tot = d.sum(units)
    q.put((rank, mx, tot, bench.aggregate(tot, mx)))
    d.close()


def test_weak_scaling_bookkeeping_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, mx, tot, val in res:
        assert mx == 2.0 and tot == 24.0 and val == pytest.approx(12.0)


def test_aggregate_single_rank():
    import bench
    assert bench.aggregate(80.0, 2.0) == 40.0


def test_summarize_takes_the_median_repeat_and_its_spread():
    import bench
    times = [0.010, 0.012, 0.011, 0.030, 0.011]  # seconds per repeat of K = 10 steps; one outlier
    r = bench.summarize(times, units=80.0, K=10, path_bytes=1e6, peak=1000.0)
    assert r["value"] == pytest.approx(80.0 / 0.011)
    assert r["ms_per_step"] == pytest.approx(1.1)
    assert r["achieved_gbs"] == pytest.approx(1e6 * 10 / 0.011 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved_gbs"] / 1000.0)
    assert r["repeats"]["n"] == 5
    assert r["repeats"]["min_value"] == pytest.approx(80.0 / 0.030)
    assert r["repeats"]["spread"] == pytest.approx((0.030 - 0.010) / 0.011)

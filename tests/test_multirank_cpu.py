"""The N > 1 host logic of bench.py on CPU: two gloo ranks (127.0.0.1).

Each rank re-scores an independent workload (its own seed; weak scaling, no
collective on the data path); the ranks meet at barriers around the timed
region and the job time is the maximum over ranks."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist

    import bench
    w, r, _ = bench.dist_setup()
    assert dist.get_backend() == "gloo" and w == world and r == rank
    bench.barrier(w)
    t = bench.max_over_ranks(100.0 + 50.0 * rank, w)     # per-rank step times in ms
    spec = bench.spec_for("math", seed=r)
    # rank 1 alone saw a thermal slowdown: both ranks must take the timing again
    clk = {"sm_mhz": 1900.0, "sm_max_mhz": 2070.0,
           "reasons": ["sw_thermal_slowdown"] if r == 1 else []}
    again = bench.max_over_ranks(float(bench.clock_suspect(clk)), w) > 0
    q.put((r, t, spec.seed, bench.aggregate_value(w, 1000, 10, t), again))
    bench.barrier(w)
    dist.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        res = sorted(q.get(timeout=180) for _ in procs)
    finally:
        for p in procs:
            p.join(timeout=60)
    assert all(p.exitcode == 0 for p in procs)
    assert [x[1] for x in res] == [150.0, 150.0]          # slowest rank's time
    assert [x[2] for x in res] == [0, 1]                  # independent workloads
    assert res[0][3] == pytest.approx(2 * 1000 * 10 / 0.150)
    assert [x[4] for x in res] == [True, True]            # re-measured on every rank


def test_aggregate_value_single_rank():
    import bench
    assert bench.aggregate_value(1, 155979, 10, 2000.0) == pytest.approx(779895.0)


def test_clock_suspect_rules():
    import bench
    ok = dict(sm_mhz=1580.0, sm_max_mhz=2070.0)
    assert not bench.clock_suspect(dict(ok, reasons=["sw_power_cap"]))      # kept and noted
    assert not bench.clock_suspect(dict(sm_mhz=2070.0, sm_max_mhz=2070.0, reasons=[]))
    for r in bench.SLOWDOWNS:
        assert bench.clock_suspect(dict(ok, reasons=[r, "sw_power_cap"]))
    assert bench.clock_suspect(dict(ok, reasons=[]))      # low clock, no reason: a lock
    assert not bench.clock_suspect({"sm_mhz": None, "sm_max_mhz": None,
                                    "reasons": ["nvidia-smi unavailable"]})

"""Multi-rank logic on CPU with two gloo ranks (127.0.0.1).

bench.py at N > 1: each rank re-scores an independent workload (its own seed;
weak scaling, no collective on the data path); the ranks meet at barriers
around the timed region and the job time is the maximum over ranks.

The vocabulary-parallel LM head: each rank's shard statistics, one
all-gather, and the merge, against the unsharded oracle."""
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


def _shard_worker(rank, world, port, q):
    """One rank of a vocabulary-parallel LM head: its own columns of W, the
    per-row statistics of its shard (max, sum of exponentials, the target's
    logit if this shard owns the target column, the p-weighted logit sum),
    one all-gather of those statistics (the only exchange), then the merge
    every rank performs locally."""
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    import numpy as np
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    rng = np.random.default_rng(11)                     # same draw on every rank
    n, d, V = 37, 24, 101
    h = rng.normal(size=(n, d))
    w = rng.normal(size=(V, d)) * 0.7
    y = rng.integers(0, V, size=n)
    cuts = [0, 40, V] if world == 2 else [0, V]
    lo, hi = cuts[rank], cuts[rank + 1]
    z = h @ w[lo:hi].T                                  # this shard's logits only
    m = z.max(axis=1)
    e = np.exp(z - m[:, None])
    s = e.sum(axis=1)
    own = (y >= lo) & (y < hi)
    zt = np.where(own, z[np.arange(n), np.clip(y - lo, 0, hi - lo - 1)], np.nan)
    t = (e * z).sum(axis=1)
    mine = torch.from_numpy(np.stack([m, s, zt, t], axis=1))    # [n, 4]
    got = [torch.empty_like(mine) for _ in range(world)]
    dist.all_gather(got, mine)
    st = torch.stack(got).numpy()                       # [P, n, 4]
    M = st[:, :, 0].max(axis=0)
    scale = np.exp(st[:, :, 0] - M)
    S = (st[:, :, 1] * scale).sum(axis=0)
    T = (st[:, :, 3] * scale).sum(axis=0)
    Z = np.nanmax(st[:, :, 2], axis=0)                  # exactly one shard owns each target
    logp = Z - M - np.log(S)
    ent = M + np.log(S) - T / S
    q.put((rank, logp, ent, int(np.isnan(st[:, :, 2]).sum())))
    dist.destroy_process_group()


def test_vocab_sharded_exchange_two_gloo_ranks():
    """The vocabulary-parallel LM head's exchange on two CPU ranks: after one
    all-gather of 4 statistics per row and shard, every rank's merged log-probs
    and entropies equal the unsharded oracle's."""
    import numpy as np
    import oracle
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        res = sorted((q.get(timeout=180) for _ in procs), key=lambda x: x[0])
    finally:
        for p in procs:
            p.join(timeout=60)
    assert all(p.exitcode == 0 for p in procs)
    rng = np.random.default_rng(11)
    n, d, V = 37, 24, 101
    h = rng.normal(size=(n, d))
    w = rng.normal(size=(V, d)) * 0.7
    y = rng.integers(0, V, size=n)
    ref_lp = oracle.target_logprobs(h, w, y)
    ref_h = oracle.next_token_entropy(h, w)
    for rank, logp, ent, n_missing in res:
        assert n_missing == n                           # each target owned by one shard
        assert np.allclose(logp, ref_lp, rtol=0, atol=1e-12)
        assert np.allclose(ent, ref_h, rtol=0, atol=1e-12)

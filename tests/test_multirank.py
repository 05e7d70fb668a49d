"""Multi-rank host logic on CPU with gloo process groups (world size 2 and 4):
the bench's whole-job reduction and the foreground-count bucketing schedule
that data-parallel replicas follow without exchanging it."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_23169_gb300 import bucketing as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _counts(n=103, seed=0):
    """Foreground token counts of n samples: 13 images of 16,384 tokens at a
    foreground fraction of 5-51% (the paper's range) per sample."""
    g = np.random.Generator(np.random.PCG64(seed))
    return np.rint(13 * 16384 * g.uniform(0.05, 0.512, size=n)).astype(np.int64)


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import sys
        sys.path.insert(0, ROOT)
        import bench
        # whole-job: slowest rank's time, summed work
        ms, fl = bench.whole_job(10.0 + rank, 1e12 * (rank + 1), world, "cpu")
        # bucketing: every rank builds the schedule alone and takes its column
        counts = _counts()
        mine = B.rank_samples(counts, world, rank, seed=3, epoch=1)
        gathered = [torch.zeros(len(mine), dtype=torch.int64) for _ in range(world)]
        dist.all_gather(gathered, torch.from_numpy(mine))
        q.put((rank, ms, fl, [g.numpy() for g in gathered]))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 4])
def test_gloo_ranks_agree(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=240) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    want_ms, want_fl = 10.0 + world - 1, 1e12 * world * (world + 1) / 2
    sched = B.fg_schedule(_counts(), world, seed=3, epoch=1)
    for rank, ms, fl, cols in res:
        assert ms == want_ms and fl == want_fl
        # the columns the ranks took are exactly the schedule built on one host
        assert np.array_equal(np.stack(cols, axis=1), sched)


def test_schedule_covers_the_epoch_and_balances():
    counts = _counts(1003, seed=1)
    for world in (1, 2, 8, 64):
        s = B.fg_schedule(counts, world, seed=0, epoch=0)
        n = len(counts)
        assert s.shape == (-(-n // world), world)
        ids, reps = np.unique(s, return_counts=True)
        assert np.array_equal(ids, np.arange(n))                 # every sample in the epoch
        assert reps.sum() - n == s.size - n < world               # repeats only to fill the last step
        if world > 1:
            imb = B.step_imbalance(counts, s)
            g = np.random.Generator(np.random.PCG64(5))
            rnd = g.permutation(np.resize(np.arange(n), s.size)).reshape(s.shape)
            rnd_imb = B.step_imbalance(counts, rnd).mean()
            # a step holds `world` neighbours of the sorted counts: near-perfect
            # for small worlds, and always far better than a random assignment
            assert imb.mean() < (1.05 if world <= 8 else 1.25) and imb.mean() - 1 < 0.25 * (rnd_imb - 1)
    # deterministic per (seed, epoch); another epoch reorders
    a = B.fg_schedule(counts, 8, seed=2, epoch=4)
    assert np.array_equal(a, B.fg_schedule(counts, 8, seed=2, epoch=4))
    assert not np.array_equal(a, B.fg_schedule(counts, 8, seed=2, epoch=5))
    # no rank always gets its step's longest sample
    longest = np.argmax(counts[a], axis=1)
    assert len(np.unique(longest)) == 8
    assert B.fg_schedule([], 4).shape == (0, 4)

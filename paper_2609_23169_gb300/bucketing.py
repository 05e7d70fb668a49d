"""Foreground-count bucketing of training samples across data-parallel replicas.

The paper trains with one sample per GPU and buckets the samples by their
effective foreground token count, so that the GPUs of one data-parallel step
process sequences of similar length (Sec. 4.1, training details).  With
background token dropping every sample has its own sequence length N, and the
attention cost grows with N^2 at a fixed density: an unbalanced step waits
for its longest sample.

``fg_schedule`` builds one epoch's global schedule on every rank from the same
inputs (the per-sample foreground token counts, a seed and the epoch number),
so the ranks agree without exchanging anything; rank r takes slot r of every
step.  Per epoch: a seeded permutation breaks ties between equal counts, a
stable sort by count orders the samples, consecutive runs of ``world``
samples form the steps (neighbours in the sorted order have the closest
lengths), the order of the steps is shuffled (so an epoch does not run from
the shortest to the longest sequences) and the slots inside each step are
rotated (so no rank always draws its step's longest sample).  When the
sample count is not a multiple of ``world``, the last, partial step is
completed with repeats of its own samples.
"""
from __future__ import annotations

from typing import Sequence

import numpy as np


def fg_schedule(fg_counts: Sequence[int], world: int, seed: int = 0, epoch: int = 0) -> np.ndarray:
    """[steps, world] sample ids of one epoch; row s is global step s, column r rank r."""
    counts = np.asarray(fg_counts, dtype=np.int64)
    if world < 1:
        raise ValueError("world must be >= 1")
    n = counts.size
    if n == 0:
        return np.zeros((0, world), dtype=np.int64)
    g = np.random.Generator(np.random.PCG64([int(seed), int(epoch), 0x5eed]))
    perm = g.permutation(n)
    order = perm[np.argsort(counts[perm], kind="stable")]
    steps = -(-n // world)
    pad = steps * world - n
    if pad:
        tail = order[n - (world - pad):]                     # the partial step's own samples
        order = np.concatenate([order, tail[np.arange(pad) % tail.size]])
    sched = order.reshape(steps, world)
    sched = sched[g.permutation(steps)]
    shifts = g.integers(0, world, size=steps)
    rows = np.arange(world)[None, :]
    return np.take_along_axis(sched, (rows + shifts[:, None]) % world, axis=1)


def rank_samples(fg_counts: Sequence[int], world: int, rank: int, seed: int = 0, epoch: int = 0) -> np.ndarray:
    """The sample ids rank ``rank`` processes in this epoch, one per global step."""
    if not 0 <= rank < world:
        raise ValueError("rank out of range")
    return fg_schedule(fg_counts, world, seed, epoch)[:, rank]


def step_imbalance(fg_counts: Sequence[int], schedule: np.ndarray, cost_power: float = 2.0) -> np.ndarray:
    """Per step: the slowest rank's cost over the mean rank cost, with cost
    N^cost_power (2 for attention at a fixed density).  1.0 is perfect balance."""
    c = np.asarray(fg_counts, dtype=np.float64)[schedule] ** cost_power
    return c.max(axis=1) / np.maximum(c.mean(axis=1), 1e-30)

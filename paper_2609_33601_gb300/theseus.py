"""Stage-1 schedule of Theseus QAD (Sec. 3, "Stage 1"; Algorithm 1; Table 1): which
distillation widths the student is trained at, and how many of the T1 Stage-1 steps each
width gets.  Host logic only: it decides the training loop's order, not any arithmetic on
tensors.

Widths (BinaryMergeWidths).  Start from L one-block segments and merge neighbouring segments in
pairs, level after level, until one segment spans the model; a level with an odd count carries
its last segment up unmerged.  A level's width is its widest segment, so a 28-block DiT gets
(1, 2, 4, 8, 16, 28), the widths the paper lists, and every block lies in exactly one segment of
every level (at L = 28 the last segments of levels 3 and 4 span 4 and 12 blocks).

Budget (Allocate).  Level k gets N_k steps with N_k proportional to gamma^k and sum N_k = T1
(Sec. 3), as integers: each level first takes the integer part of its exact quota, and the steps
left over go one each to the levels with the largest fractional parts, ties to the lower level.
gamma = 0 and gamma = inf are the endpoint schedules, all T1 steps at the first or the last
level.  This rule reproduces every allocation Table 1 prints (its "0.33" row is gamma = 1/3).
"""
from __future__ import annotations

import math
from fractions import Fraction

__all__ = ["binary_merge_segments", "binary_merge_widths", "allocate", "stage_one_schedule"]


def binary_merge_segments(L: int) -> list[list[tuple[int, int]]]:
    """Per level, the (first block, number of blocks) of each segment, shortest level first."""
    if L < 1:
        raise ValueError(f"the model needs at least one block, got L = {L}")
    levels = [[(b, 1) for b in range(L)]]
    while len(levels[-1]) > 1:
        prev = levels[-1]
        merged = [(prev[i][0], prev[i][1] + prev[i + 1][1]) for i in range(0, len(prev) - 1, 2)]
        if len(prev) % 2:
            merged.append(prev[-1])
        levels.append(merged)
    return levels


def binary_merge_widths(L: int) -> tuple[int, ...]:
    """(w_0, ..., w_K): the widest segment of each level."""
    return tuple(max(w for _, w in level) for level in binary_merge_segments(L))


def allocate(T1: int, gamma, levels: int) -> tuple[int, ...]:
    """Integer step counts (N_0, ..., N_{levels-1}) with N_k proportional to gamma^k, summing to T1.

    gamma may be an int, a float, a Fraction (exact quotas), 0 or math.inf.  Quotas are formed
    exactly from the value given (a float is taken at its binary value)."""
    if T1 < 0 or levels < 1:
        raise ValueError(f"need T1 >= 0 and at least one level, got T1 = {T1}, levels = {levels}")
    if gamma == 0:
        return (T1,) + (0,) * (levels - 1)
    if gamma == math.inf:
        return (0,) * (levels - 1) + (T1,)
    g = Fraction(gamma)
    if g < 0:
        raise ValueError(f"gamma must be >= 0, got {gamma}")
    weights = [g ** k for k in range(levels)]
    total = sum(weights)
    quotas = [T1 * w / total for w in weights]
    counts = [math.floor(q) for q in quotas]
    left = T1 - sum(counts)
    by_remainder = sorted(range(levels), key=lambda k: (-(quotas[k] - counts[k]), k))
    for k in by_remainder[:left]:
        counts[k] += 1
    return tuple(counts)


def stage_one_schedule(L: int, T1: int, gamma) -> list[dict]:
    """One entry per level, shortest first: its width, its steps and its segments.  Levels with
    no steps stay in the list (the training loop skips them)."""
    segments = binary_merge_segments(L)
    steps = allocate(T1, gamma, len(segments))
    return [{"level": k, "width": max(w for _, w in seg), "steps": n, "segments": seg}
            for k, (seg, n) in enumerate(zip(segments, steps))]

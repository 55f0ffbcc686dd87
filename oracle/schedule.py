"""Brute-force makespan search over schedules of a small GEMM set —
TEST INFRASTRUCTURE ONLY.

What it computes.  The paper's "Oracle" configuration uses the GO-Kernels and
always picks the right concurrency degree, sequential execution included
(Sec. 5.5, Configurations).  For a set of n independent GEMMs, a schedule is
written here as an ordered split of the set into groups that run one after
another; the GEMMs inside a group run concurrently, so the group's
concurrency degree (CD) is its size; each GEMM runs one kernel variant chosen
from an allowed list.  The makespan of a schedule is the sum of its groups'
times, and a group's time is read from a timing table supplied by the caller
(measured once on the GPU, or synthetic in unit tests).  Every set partition
of the n GEMMs and every variant choice is enumerated; the search returns the
minimum, ties broken by (fewer groups, smaller largest CD, lexicographically
smaller variant tuple, lexicographically smaller partition).

The order of groups does not change a sum, so a partition is enumerated once,
in canonical form (blocks sorted by their smallest member).  The number of
partitions of n items is the Bell number B(n) (1, 1, 2, 5, 15, 52, 203, ...),
which the tests check.

``subset_dp`` computes the same optimum by a different algorithm (dynamic
programming over subsets), to pin the enumeration.
"""
from __future__ import annotations

import itertools
from dataclasses import dataclass
from typing import Callable, Dict, Iterator, List, Sequence, Tuple

Block = Tuple[int, ...]
Partition = Tuple[Block, ...]


def set_partitions(n: int) -> Iterator[Partition]:
    """Every partition of {0..n-1}, blocks in increasing order of their
    smallest element, members sorted.  Built from restricted growth strings:
    item i joins one of the blocks opened so far or opens a new one."""
    if n == 0:
        yield ()
        return
    labels = [0] * n

    def rec(i: int, n_blocks: int):
        if i == n:
            blocks: List[List[int]] = [[] for _ in range(n_blocks)]
            for item, lab in enumerate(labels):
                blocks[lab].append(item)
            yield tuple(tuple(b) for b in blocks)
            return
        for lab in range(n_blocks + 1):
            labels[i] = lab
            yield from rec(i + 1, max(n_blocks, lab + 1))

    labels[0] = 0
    yield from rec(1, 1)


def bell_number(n: int) -> int:
    """B(n) from the Bell triangle (independent of the enumeration above)."""
    if n == 0:
        return 1
    row = [1]
    for _ in range(n - 1):
        nxt = [row[-1]]
        for v in row:
            nxt.append(nxt[-1] + v)
        row = nxt
    return row[-1]


ChoicesFn = Callable[[int, Block], Sequence[int]]
GroupTimeFn = Callable[[Block, Tuple[int, ...]], float]


@dataclass(frozen=True)
class Best:
    makespan: float
    partition: Partition
    variants: Tuple[int, ...]      # variant of GEMM i, indexed by i

    @property
    def n_groups(self) -> int:
        return len(self.partition)

    @property
    def max_cd(self) -> int:
        return max((len(b) for b in self.partition), default=0)


def brute_force(n: int, choices: ChoicesFn, group_time: GroupTimeFn) -> Best:
    """Exhaustive minimum-makespan schedule.

    ``choices(i, block)`` lists the variants GEMM i may run with when it runs
    concurrently with the members of ``block`` (a GEMM library returns kernels
    per CD, Sec. 4.2.2).  ``group_time(block, variants)`` is the time of running
    ``block`` concurrently, ``variants[j]`` being the variant of ``block[j]``.
    """
    best_key = None
    best = None
    for part in set_partitions(n):
        per_block = []
        for blk in part:
            per_block.append([tuple(v) for v in
                              itertools.product(*[list(choices(i, blk)) for i in blk])])
        for combo in itertools.product(*per_block):
            total = 0.0
            variants = [0] * n
            for blk, vs in zip(part, combo):
                total += float(group_time(blk, vs))
                for i, v in zip(blk, vs):
                    variants[i] = v
            vt = tuple(variants)
            key = (total, len(part), max(len(b) for b in part) if part else 0, vt, part)
            if best_key is None or key < best_key:
                best_key = key
                best = Best(total, part, vt)
    if best is None:
        return Best(0.0, (), ())
    return best


def subset_dp(n: int, choices: ChoicesFn, group_time: GroupTimeFn) -> float:
    """Optimal makespan by dynamic programming over subsets: the cheapest way
    to finish subset S is the cheapest block T containing the smallest member
    of S plus the cheapest way to finish S without T."""
    full = (1 << n) - 1
    block_cost: Dict[int, float] = {}
    for mask in range(1, full + 1):
        blk = tuple(i for i in range(n) if mask >> i & 1)
        best = None
        for vs in itertools.product(*[list(choices(i, blk)) for i in blk]):
            t = float(group_time(blk, tuple(vs)))
            if best is None or t < best:
                best = t
        block_cost[mask] = best
    f = {0: 0.0}
    for mask in range(1, full + 1):
        low = mask & -mask
        rest = mask ^ low
        best = None
        sub = rest
        while True:
            t_mask = sub | low
            v = block_cost[t_mask] + f[mask ^ t_mask]
            if best is None or v < best:
                best = v
            if sub == 0:
                break
            sub = (sub - 1) & rest
        f[mask] = best
    return f[full]


def makespan_of(partition: Partition, variants: Sequence[int], group_time: GroupTimeFn) -> float:
    """Makespan of one given schedule under the same timing table."""
    total = 0.0
    for blk in partition:
        total += float(group_time(tuple(blk), tuple(variants[i] for i in blk)))
    return total

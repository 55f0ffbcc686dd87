"""Pins for the brute-force schedule search (CPU only): Bell numbers,
hand-solved timing tables, tie-breaking, and agreement with an independent
dynamic program over subsets."""
import itertools
import random

import pytest

from oracle import schedule as sch

# B(0..8), as tabulated in the literature (OEIS A000110)
BELL = [1, 1, 2, 5, 15, 52, 203, 877, 4140]


@pytest.mark.parametrize("n", range(0, 8))
def test_partition_count_is_bell(n):
    parts = list(sch.set_partitions(n))
    assert len(parts) == BELL[n] == sch.bell_number(n)
    seen = set()
    for p in parts:
        items = [i for blk in p for i in blk]
        assert sorted(items) == list(range(n))           # cover, disjoint
        assert all(list(b) == sorted(b) for b in p)
        assert [b[0] for b in p] == sorted(b[0] for b in p)
        seen.add(p)
    assert len(seen) == len(parts)                        # no repeats


def _table_from(d):
    def gt(block, variants):
        return d[(tuple(block), tuple(variants))]
    return gt


def test_two_gemms_concurrency_wins():
    # each alone takes 1.0; together 1.5 -> run concurrently (makespan 1.5)
    d = {((0,), (0,)): 1.0, ((1,), (0,)): 1.0, ((0, 1), (0, 0)): 1.5}
    best = sch.brute_force(2, lambda i, b: [0], _table_from(d))
    assert best.partition == ((0, 1),) and best.makespan == 1.5


def test_two_gemms_sequential_wins():
    # contention makes the pair slower than running them back to back
    d = {((0,), (0,)): 1.0, ((1,), (0,)): 1.0, ((0, 1), (0, 0)): 2.5}
    best = sch.brute_force(2, lambda i, b: [0], _table_from(d))
    assert best.partition == ((0,), (1,)) and best.makespan == 2.0


def test_tie_prefers_fewer_groups():
    d = {((0,), (0,)): 1.0, ((1,), (0,)): 1.0, ((0, 1), (0, 0)): 2.0}
    best = sch.brute_force(2, lambda i, b: [0], _table_from(d))
    assert best.partition == ((0, 1),)


def test_variant_choice_depends_on_group():
    # variant 7 is the isolated kernel, variant 9 the kernel tuned for CD 2:
    # alone 7 is faster, together the 9/9 pair is best.
    def choices(i, blk):
        return [7, 9]
    t = {}
    for i in (0, 1):
        t[((i,), (7,))] = 1.0
        t[((i,), (9,))] = 1.3
    for v in itertools.product([7, 9], repeat=2):
        t[((0, 1), v)] = {(7, 7): 2.4, (7, 9): 1.9, (9, 7): 1.9, (9, 9): 1.6}[v]
    best = sch.brute_force(2, choices, _table_from(t))
    assert best.partition == ((0, 1),) and best.variants == (9, 9)
    assert best.makespan == pytest.approx(1.6)


def test_three_gemms_hand_solved():
    # G0 and G1 overlap well, G2 hurts anything it runs with.
    def gt(block, variants):
        s = set(block)
        if s == {0} or s == {1}:
            return 1.0
        if s == {2}:
            return 2.0
        if s == {0, 1}:
            return 1.2
        return 10.0                                       # any group holding 2 with others
    best = sch.brute_force(3, lambda i, b: [0], gt)
    assert best.partition == ((0, 1), (2,))
    assert best.makespan == pytest.approx(3.2)


@pytest.mark.parametrize("seed", range(12))
def test_brute_force_equals_subset_dp(seed):
    rng = random.Random(seed)
    n = rng.randint(1, 5)
    table = {}

    def choices(i, blk):
        return [0, 1] if len(blk) > 1 else [0]

    def gt(block, variants):
        key = (tuple(block), tuple(variants))
        if key not in table:
            table[key] = rng.uniform(0.5, 3.0) * (0.6 + 0.4 * len(block))
        return table[key]

    best = sch.brute_force(n, choices, gt)
    dp = sch.subset_dp(n, choices, gt)
    assert best.makespan == pytest.approx(dp, rel=1e-12)
    assert sch.makespan_of(best.partition, best.variants, gt) == pytest.approx(best.makespan)

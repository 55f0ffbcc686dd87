"""goldy_plan (C++) against the independent Python restatement in
oracle/planner_ref.py: byte-identical schedules on 10^4 random descriptor
sets and random lookup tables, every policy, and determinism."""
import random

import pytest

from oracle import planner_ref as pr
from paper_2409_02227_gb300 import goldy as G

NV = 120


def random_lut(rng, n_entries):
    keys = set()
    while len(keys) < n_entries:
        keys.add((rng.randint(3, 13), rng.randint(7, 14), rng.randint(7, 14), rng.randint(0, 1)))
    entries = [pr.Entry(k, rng.choice(pr.CD_CLASSES), tuple(rng.randrange(NV) for _ in range(5)))
               for k in keys]
    return pr.write_lut(entries, NV)


def random_desc(rng, shapes):
    if shapes and rng.random() < 0.6:
        return rng.choice(shapes)
    M = rng.choice([rng.randint(1, 5000), rng.choice([16, 32, 128, 512, 2048, 4096])])
    N = 64 * rng.randint(1, 130)
    K = 64 * rng.randint(1, 130)
    return (M, N, K, rng.randint(0, 1))


def flags_for(rng):
    pol = rng.choice([0, 0, 0, 0, 1, 2, 3, 4])
    if pol == 4:
        pol |= rng.randint(1, 20) << 8
    if rng.random() < 0.3:
        pol |= G.GOLDY_PLAN_FUSED
    return pol


@pytest.mark.parametrize("chunk", range(10))
def test_random_sets_byte_identical(chunk):
    rng = random.Random(1234 + chunk)
    for trial in range(1000):
        lut_bytes = random_lut(rng, rng.randint(1, 40))
        lut = G.goldy_lut_from_memory(lut_bytes)
        shapes = []
        n = rng.choice([1, 2, 3, 4, 5, 8, 16, rng.randint(1, 64)])
        descs = []
        for _ in range(n):
            t = random_desc(rng, shapes)
            shapes.append(t)
            descs.append(t)
        flags = flags_for(rng)
        ref = pr.serialize(pr.plan([pr.Desc(*t) for t in descs], lut_bytes, flags))
        gd = [G.desc(M, N, K, c) for (M, N, K, c) in descs]
        got = G.goldy_serialize = G.goldy_schedule_serialize(G.goldy_plan(gd, lut, flags))
        assert got == ref, (trial, descs, flags)


def test_deterministic():
    rng = random.Random(7)
    lut_bytes = random_lut(rng, 30)
    lut = G.goldy_lut_from_memory(lut_bytes)
    descs = [G.desc(*random_desc(rng, [])) for _ in range(12)]
    first = G.goldy_schedule_serialize(G.goldy_plan(descs, lut))
    for _ in range(20):
        assert G.goldy_schedule_serialize(G.goldy_plan(descs, lut)) == first
    lut2 = G.goldy_lut_from_memory(lut_bytes)
    assert G.goldy_schedule_serialize(G.goldy_plan(descs, lut2)) == first


def test_config_sets_against_reference():
    from paper_2409_02227_gb300 import workloads as wl
    rng = random.Random(11)
    lut_bytes = random_lut(rng, 60)
    lut = G.goldy_lut_from_memory(lut_bytes)
    sets = [wl.config_specs(n)[1] for n in wl.FIXED_CONFIGS]
    sets += [wl.sweep_specs(j)[1] for j in range(64)]
    for specs in sets:
        for flags in (0, 1, 2, 3, G.force_cd(2), G.force_cd(4)):
            ref = pr.serialize(pr.plan([pr.Desc(s.M, s.N, s.K, s.out_dtype) for s in specs], lut_bytes, flags))
            got = G.goldy_schedule_serialize(
                G.goldy_plan([G.desc(s.M, s.N, s.K, s.out_dtype) for s in specs], lut, flags))
            assert got == ref

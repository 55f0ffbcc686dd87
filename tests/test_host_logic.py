"""Host-side logic that needs no GPU: the profiler's preferred-CD rule and LUT
writer against the oracle's independent versions, and bench.py's multi-rank
aggregation (barrier + max over ranks) on world_size-2 gloo process groups."""
import os
import random
import socket

import pytest
import torch.multiprocessing as mp

from oracle import planner_ref as pr
from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import profile_lut as P


def test_preferred_cd_matches_oracle():
    rng = random.Random(5)
    for _ in range(5000):
        sp = {1: 1.0}
        for cd in (2, 4, 8, 16):
            if rng.random() < 0.9:
                sp[cd] = rng.choice([rng.uniform(0.5, 2.5), rng.uniform(0.98, 1.08)])
        assert P.preferred_cd(sp) == pr.preferred_cd(sp), sp
    # a CD within 1% of the best does not win: the largest speedup does
    for sp in ({1: 1.0, 2: 1.20, 4: 1.195}, {1: 1.0, 4: 2.126, 8: 2.111}, {1: 1.0, 8: 1.658, 16: 1.647}):
        assert P.preferred_cd(sp) == pr.preferred_cd(sp) == max(sp, key=sp.get)


def test_table_preferences_follow_the_logged_speedups():
    """The packaged table's preferred CDs are the rule applied to the
    speedups its profiling log recorded."""
    import json
    import struct
    data = open(G.DEFAULT_LUT, "rb").read()
    n = struct.unpack_from("<I", data, 12)[0]
    prefs = {tuple(data[32 + 16 * i:32 + 16 * i + 4]): data[32 + 16 * i + 4] for i in range(n)}
    log = os.path.join(os.path.dirname(G.DEFAULT_LUT), "lut_profile.jsonl")
    for line in open(log):
        r = json.loads(line)
        sp = {int(c): v for c, v in r["speedup"].items()}
        assert prefs[tuple(r["key"])] == pr.preferred_cd(sp), r["key"]


def test_lut_writer_matches_oracle_format():
    rng = random.Random(9)
    keys = {(rng.randint(3, 13), rng.randint(7, 14), rng.randint(7, 14), rng.randint(0, 1)) for _ in range(50)}
    entries = [(k, rng.choice(pr.CD_CLASSES), [rng.randrange(120) for _ in range(5)]) for k in keys]
    mine = P.write_lut(entries, 120, 152)
    ref = pr.write_lut([pr.Entry(k, p, tuple(v)) for k, p, v in entries], 120, 152)
    assert mine == ref
    G.goldy_lut_from_memory(mine)
    # with the co-run flag of step 3
    flagged = [(k, p, v, rng.randint(0, 3) | (rng.randint(0, 2) << 2)) for k, p, v in entries]
    mine = P.write_lut(flagged, 120, 152)
    assert mine == pr.write_lut([pr.Entry(k, p, tuple(v), f) for k, p, v, f in flagged], 120, 152)
    G.goldy_lut_from_memory(mine)


def test_bucket_shapes_and_candidates():
    assert P.bucket_shape((7, 10, 12, 0)) == (128, 1024, 4096, 0)
    # centre 2^(l + 1/2): 128 * sqrt2 = 181.02, 1024 * sqrt2 = 1448.2 -> 64 * 23, 4096 * sqrt2 = 5792.6 -> 64 * 91
    assert P.bucket_centre((7, 10, 12, 0)) == (181, 1472, 5824, 0)
    assert P.bucket_points((7, 10, 12, 0)) == [(128, 1024, 4096, 0), (181, 1472, 5824, 0)]
    # every centre lies inside its bucket
    for key in [(4, 8, 9, 1), (11, 13, 11, 0), (6, 12, 8, 1)]:
        M, N, K, _ = P.bucket_centre(key)
        assert (M.bit_length() - 1, N.bit_length() - 1, K.bit_length() - 1) == key[:3]
    c = P.candidates(32, 4096, 1024, 152)
    kinds = {k for k, _ in c}
    assert {6, 7, 8, 9} <= kinds                      # transposed tiles offered for skinny M
    assert all(s in (1, 2, 4, 8) for _, s in c)
    big = {k for k, _ in P.candidates(512, 1024, 1024, 152)}
    assert not {6, 7, 8, 9} & big and 10 in big
    # the pair kind splits K too: 2 x 4 tiles of 256 x 256, K = 1024 -> 16 blocks
    assert sorted(s for k, s in P.candidates(512, 1024, 1024, 152) if k == 10) == [1, 2, 4, 8]
    # ...but not beyond the K blocks (K = 128: 2 blocks) or 4 x the SMs of units
    assert sorted(s for k, s in P.candidates(512, 1024, 128, 152) if k == 10) == [1, 2]
    assert sorted(s for k, s in P.candidates(4096, 8192, 4096, 152) if k == 10) == [1]


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, l = bench.dist_env()
    dist = bench.dist_init(w, "gloo")
    bench.barrier(dist)
    got = bench.reduce_max(10.0 + rank, dist)
    q.put((r, got))
    dist.destroy_process_group()


def test_multi_rank_max_over_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res == {0: 11.0, 1: 11.0}


def test_corun_flags_rule():
    base = {"sequential": 10.0, "v0_rc1": 9.9, "v0_rc2": 9.8, "v0_rc4": 9.7, "v1_rc1": 9.6, "v1_rc2": 9.9,
            "v1_rc4": 9.9}
    assert P.corun_flags(base) == 0                       # nothing at once gains 5% over one after the other
    t = dict(base, v0_rc1=9.0)
    assert P.corun_flags(t) == 0b0001                     # the default configuration at once
    t = dict(base, v0_rc1=9.0, v1_rc2=8.8)
    assert P.corun_flags(t) == 0b0001                     # 8.8 is not 5% better than the default's 9.0
    t = dict(base, v0_rc1=9.0, v1_rc2=8.0)
    assert P.corun_flags(t) == 0b0111                     # CD-2 kernel, op at GPU/2
    t = dict(base, v0_rc1=9.0, v0_rc4=7.0, v1_rc2=7.0)
    assert P.corun_flags(t) == 0b0111                     # ties: the smaller flag word
    t = dict(base, v0_rc1=12.0, v0_rc4=9.0)
    assert P.corun_flags(t) == 0b1001
    # every configuration the table can record round-trips through the planner
    import random as _r
    from oracle import planner_ref as pr
    for name, flags in P.CORUN_CONFIGS:
        lut = P.write_lut([((7, 10, 12, 0), 4, [10, 11, 12, 13, 14], flags)], 132, 152)
        conc, v, rc = pr.corun_plan(pr.Desc(128, 1024, 4096, 0), lut, pr.POLICY_AUTO)
        assert conc == 1 and v == (11 if name.startswith("v1") else 10) and rc == int(name.split("rc")[1])


def test_pick_variant_scores_relative_times():
    # one point: the fastest wins
    assert P.pick_variant({3: [10.0], 7: [9.0], 5: [9.5]}) == 7
    # two points: 7 is fastest at the first point by 1%, but 40% off at the
    # second; 3 is 5% off at the first and fastest at the second -> 3
    assert P.pick_variant({3: [10.5, 20.0], 7: [10.0, 28.0]}) == 3
    # relative, not absolute: a 1 us point and a 100 us point weigh the same
    # (mean ratios 1.10 vs 1.15; summed times would pick 2: 121 vs 101.3 us)
    assert P.pick_variant({1: [1.0, 120.0], 2: [1.3, 100.0]}) == 1
    # ties -> smaller id
    assert P.pick_variant({9: [2.0, 4.0], 4: [2.0, 4.0]}) == 4


def test_rank_variants_orders_by_relative_time():
    # mean ratio to the fastest at each point: 7 (1.0, 1.4) -> 1.2; 3 (1.05, 1.0)
    # -> 1.025; 5 (1.1, 1.2) -> 1.15; ties to the smaller id
    times = {3: [10.5, 20.0], 7: [10.0, 28.0], 5: [11.0, 24.0], 2: [11.0, 24.0]}
    assert P.rank_variants(times) == [3, 2, 5, 7]
    assert P.pick_variant(times) == P.rank_variants(times)[0]

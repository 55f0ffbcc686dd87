"""Pins for the reference planner (CPU only): hand-solved cases of the rules
it restates — min(preferred CD, available) (Sec. 4.3), the heterogeneous
all-or-homogeneous-groups rule (Sec. 6.7), the >= 5% sequential rule
(Sec. 5.5) — plus the LUT and schedule byte formats written out by hand."""
import struct

import pytest

from oracle import planner_ref as pr

NV = 120


def lut(*entries):
    return pr.write_lut([pr.Entry(k, p, tuple(v)) for k, p, v in entries], NV)


def D(M, N, K, out=pr.DTYPE_F32):
    return pr.Desc(M, N, K, out)


K_SMALL = (9, 10, 10, 1)          # 512 x 1024 x 1024 fp32
K_BIG = (11, 13, 11, 1)           # 2048 x 8192 x 2048 fp32
V_SMALL = (10, 11, 12, 13, 14)
V_BIG = (20, 21, 22, 23, 24)


def test_bucket_key():
    assert pr.bucket_key(256, 256, 512, 1) == (8, 8, 9, 1)
    assert pr.bucket_key(255, 257, 511, 0) == (7, 8, 8, 0)
    assert pr.bucket_key(1, 0, 4096, 0) == (0, 0, 12, 0)
    assert pr.floor_log2(2 ** 40) == 40


def test_single_gemm_runs_alone_with_isolated_kernel():
    s = pr.plan([D(512, 1024, 1024)], lut((K_SMALL, 4, V_SMALL)))
    groups, per, ms, _ = s
    assert groups == [(1, [0])] and per == [(0, 10, 0)] and ms == 1


def test_homogeneous_min_of_pref_and_available():
    L = lut((K_SMALL, 2, V_SMALL))
    groups, per, ms, _ = pr.plan([D(512, 1024, 1024)] * 4, L)
    assert groups == [(2, [0, 1, 2, 3])] and ms == 2
    assert per == [(0, 11, 0), (0, 11, 1), (0, 11, 0), (0, 11, 1)]
    # 3 available, preferred 4 -> run 3 at once with the CD-4 class kernel
    L4 = lut((K_SMALL, 4, V_SMALL))
    groups, per, ms, _ = pr.plan([D(512, 1024, 1024)] * 3, L4)
    assert groups == [(3, [0, 1, 2])] and [p[1] for p in per] == [12, 12, 12]
    assert [p[2] for p in per] == [0, 1, 2]


def test_all_prefer_sequential():
    L = lut((K_SMALL, 1, V_SMALL))
    groups, per, ms, _ = pr.plan([D(512, 1024, 1024)] * 5, L)
    assert groups == [(1, [0, 1, 2, 3, 4])] and ms == 1
    assert all(p == (0, 10, 0) for p in per)


def test_heterogeneous_pair_paper_rule():
    # 8 + 8 GEMMs of two shapes (Sec. 6.7): both prefer 16 -> all 16 at once
    L = lut((K_SMALL, 16, V_SMALL), (K_BIG, 16, V_BIG))
    descs = [D(512, 1024, 1024)] * 8 + [D(2048, 8192, 2048)] * 8
    groups, per, ms, _ = pr.plan(descs, L)
    # members listed block by block, the bigger-FLOP block first; the 16
    # run as waves of 16, so the small GEMMs take the big ones' kernel kind
    # (rule 6: variant 24 is kind 2, no split, grid-cap index 0)
    assert groups == [(16, list(range(8, 16)) + list(range(8)))] and ms == 16
    assert [p[1] for p in per] == [24] * 16
    assert per[8] == (0, 24, 0) and per[0] == (0, 24, 8)
    # one of them prefers 8 -> two homogeneous groups of 8, bigger FLOPs first
    L = lut((K_SMALL, 16, V_SMALL), (K_BIG, 8, V_BIG))
    groups, per, ms, _ = pr.plan(descs, L)
    assert groups == [(8, list(range(8, 16))), (8, list(range(8)))]
    assert per[8] == (0, 23, 0) and per[0] == (1, 23 - 10, 0)


def test_heterogeneous_three_small_one_big():
    # the mixed set from two co-running models: big prefers 1, small prefers 4
    L = lut((K_SMALL, 4, V_SMALL), (K_BIG, 1, V_BIG))
    descs = [D(512, 1024, 1024)] * 3 + [D(2048, 8192, 2048)]
    groups, per, ms, _ = pr.plan(descs, L)
    assert groups == [(1, [3]), (3, [0, 1, 2])]
    assert per[3] == (0, 20, 0)
    assert per[:3] == [(1, 12, 0), (1, 12, 1), (1, 12, 2)]
    # both prefer 4 -> all four at once
    L = lut((K_SMALL, 4, V_SMALL), (K_BIG, 4, V_BIG))
    groups, per, ms, _ = pr.plan(descs, L)
    assert groups == [(4, [3, 0, 1, 2])]
    assert per[3] == (0, 22, 0) and per[0] == (0, 12, 1)


def test_greedy_merge_many_keys():
    k1, k2, k3 = (5, 9, 9, 1), (6, 9, 9, 1), (7, 9, 9, 1)
    L = lut((k1, 4, (1, 2, 3, 4, 5)), (k2, 4, (6, 7, 8, 9, 10)), (k3, 2, (11, 12, 13, 14, 15)))
    descs = [D(32, 512, 512), D(64, 512, 512), D(128, 512, 512)]
    groups, per, ms, _ = pr.plan(descs, L)
    # FLOPs order: k3 (128 rows), k2, k1.  k3+k2 -> size 2 <= min(2, 4): merge;
    # adding k1 -> size 3 > 2: new group.  In the wave [2, 1] GEMM 1 (M = 64,
    # variant 7 = kind 0) takes GEMM 2's kind 1 (variant 12 -> 12: no split,
    # grid-cap index 0).
    assert groups == [(2, [2, 1]), (1, [0])]
    assert per == [(1, 1, 0), (0, 12, 1), (0, 12, 0)]


def vid(kind, split_idx, rc_idx):
    return (kind * 4 + split_idx) * 3 + rc_idx


def test_one_kind_per_wave_by_hand():
    # rule 6 on hand-built groups (cd, members, variants): descs M, N, K
    big = D(2048, 8192, 2048)                 # the wave's largest
    pair_v = vid(10, 0, 2)                    # CTA-pair kind, grid-cap index 2
    cases = [
        (D(512, 1024, 1024), vid(2, 1, 1), vid(10, 0, 2)),    # suits the pair kind: moved (no split, cap of the largest)
        (D(96, 1024, 1024), vid(2, 1, 1), vid(2, 1, 1)),      # M < 128: a pair kind does not suit it
        (D(512, 1024, 4096), vid(2, 1, 1), vid(2, 1, 1)),     # K longer than the largest's: kept
        (D(512, 1024, 1024, pr.DTYPE_BF16), vid(2, 1, 1), vid(2, 1, 1)),   # other output dtype: kept
        (D(512, 1024, 1024), vid(10, 0, 0), vid(10, 0, 0)),   # already the same kind: untouched
    ]
    for d, v, want in cases:
        got = pr.one_kind_per_wave([big, d], [(2, [0, 1], [pair_v, v])])
        assert got == [(2, [0, 1], [pair_v, want])], (d, v, got)
    # a transposed skinny-M kind as the largest's: only M <= 2 x 32 follows it
    t32 = vid(6, 2, 1)
    big_skinny = D(32, 8192, 4096)
    for M, want in ((64, vid(6, 0, 1)), (65, vid(0, 0, 0))):
        got = pr.one_kind_per_wave([big_skinny, D(M, 256, 512)], [(2, [0, 1], [t32, vid(0, 0, 0)])])
        assert got[0][2] == [t32, want], (M, got)
    # waves are the members taken CD at a time: with CD 1 nothing moves
    got = pr.one_kind_per_wave([big, D(512, 1024, 1024)], [(1, [0, 1], [pair_v, vid(2, 1, 1)])])
    assert got == [(1, [0, 1], [pair_v, vid(2, 1, 1)])]
    # two waves of CD 2 in launch order [0, 2, 1, 3]: each has its own
    # largest — GEMM 0 leads [0, 2]; GEMM 3 (600 rows) leads [1, 3], so GEMM
    # 1 (kind 4) takes kind 0 with GEMM 3's grid-cap index
    descs = [big, D(512, 1024, 1024), D(512, 1024, 1024), D(600, 1024, 1024)]
    got = pr.one_kind_per_wave(descs, [(2, [0, 2, 1, 3], [pair_v, vid(2, 0, 0), vid(4, 1, 0), vid(0, 0, 2)])])
    assert got == [(2, [0, 2, 1, 3], [pair_v, vid(10, 0, 2), vid(0, 0, 2), vid(0, 0, 2)])]
    # with GEMM 3's K halved, GEMM 1 leads the second wave and GEMM 3 follows it
    descs[3] = D(600, 1024, 512)
    got = pr.one_kind_per_wave(descs, [(2, [0, 2, 1, 3], [pair_v, vid(2, 0, 0), vid(4, 1, 0), vid(0, 0, 2)])])
    assert got[0][2] == [pair_v, vid(10, 0, 2), vid(4, 1, 0), vid(4, 0, 0)]
    # equal FLOPs: the first of them in launch order leads
    same = [D(512, 1024, 1024), D(512, 1024, 1024)]
    got = pr.one_kind_per_wave(same, [(2, [1, 0], [vid(2, 0, 1), vid(4, 0, 0)])])
    assert got[0][2] == [vid(2, 0, 1), vid(2, 0, 1)]


def test_nearest_key_and_ties():
    L = lut(((5, 9, 9, 1), 2, (1, 1, 1, 1, 1)), ((7, 9, 9, 1), 4, (2, 2, 2, 2, 2)))
    entries, _ = pr.parse_lut(L)
    assert pr.lookup(entries, (6, 9, 9, 1)).key == (5, 9, 9, 1)      # tie -> smaller
    assert pr.lookup(entries, (8, 9, 9, 1)).key == (7, 9, 9, 1)
    assert pr.lookup(entries, (7, 9, 9, 0)).key == (7, 9, 9, 1)      # dtype penalty only
    L2 = lut(((7, 9, 9, 0), 4, (3,) * 5), ((7, 9, 9, 1), 4, (2,) * 5))
    entries, _ = pr.parse_lut(L2)
    assert pr.lookup(entries, (7, 9, 9, 0)).key == (7, 9, 9, 0)


def test_forced_policies():
    L = lut((K_SMALL, 2, V_SMALL))
    descs = [D(512, 1024, 1024)] * 4
    g, per, ms, _ = pr.plan(descs, L, pr.POLICY_SEQUENTIAL)
    assert g == [(1, [0, 1, 2, 3])] and {p[1] for p in per} == {10}
    g, per, ms, _ = pr.plan(descs, L, pr.POLICY_DEFAULT)
    assert g == [(4, [0, 1, 2, 3])] and {p[1] for p in per} == {10} and ms == 4
    g, per, ms, _ = pr.plan(descs, L, pr.POLICY_GO)
    assert g == [(4, [0, 1, 2, 3])] and {p[1] for p in per} == {12}
    g, per, ms, _ = pr.plan(descs, L, pr.POLICY_FORCE_CD | (8 << 8))
    assert g == [(4, [0, 1, 2, 3])] and {p[1] for p in per} == {12}
    g, per, ms, _ = pr.plan(descs, L, pr.POLICY_FORCE_CD | (2 << 8))
    assert g == [(2, [0, 1, 2, 3])] and {p[1] for p in per} == {11}
    with pytest.raises(pr.PlanError):
        pr.plan(descs, L, pr.POLICY_FORCE_CD)
    with pytest.raises(pr.PlanError):
        pr.plan([], L)


def test_lut_format_by_hand():
    data = lut(((1, 2, 3, 1), 4, (5, 6, 7, 8, 9)))
    want = (b"GOLDYLUT" + struct.pack("<6I", 1, 1, NV, 0, 0, 0)
            + bytes([1, 2, 3, 1, 4, 0]) + struct.pack("<5H", 5, 6, 7, 8, 9))
    assert data == want
    with pytest.raises(pr.LutError):
        pr.parse_lut(b"GOLDYLUX" + data[8:])
    bad = bytearray(data)
    bad[32 + 6] = NV                      # variant id out of range
    with pytest.raises(pr.LutError):
        pr.parse_lut(bytes(bad))
    two = bytearray(pr.write_lut([pr.Entry((1, 2, 3, 1), 4, (0,) * 5),
                                  pr.Entry((2, 2, 3, 1), 4, (0,) * 5)], NV))
    two[32:48], two[48:64] = two[48:64], two[32:48]   # unsorted
    with pytest.raises(pr.LutError):
        pr.parse_lut(bytes(two))
    with pytest.raises(pr.LutError):
        pr.parse_lut(pr.write_lut([], NV))


def test_schedule_bytes_by_hand():
    s = ([(2, [1, 0]), (1, [2])], [(0, 5, 1), (0, 6, 0), (1, 7, 0)], 2, 0)
    words = [0x48435347, 1, 3, 2, 2, 0, 2, 2, 1, 0, 1, 1, 2, 0, 5, 1, 0, 6, 0, 1, 7, 0]
    assert pr.serialize(s) == struct.pack("<%dI" % len(words), *words)
    assert pr.serialize(s)[:4] == b"GSCH"


def test_preferred_cd_rule():
    # Sec. 4.3: the CD with the most speedup; Sec. 5.5: sequential below a 5% gain
    assert pr.preferred_cd({1: 1.0, 2: 1.04, 4: 1.049}) == 1         # below 5%
    assert pr.preferred_cd({1: 1.0, 2: 1.05}) == 2                   # exactly 5%
    assert pr.preferred_cd({1: 1.0, 2: 1.10, 4: 1.105}) == 4         # the best
    assert pr.preferred_cd({1: 1.0, 2: 1.20, 4: 1.195}) == 2         # 4 within 1% of the best: the best wins
    assert pr.preferred_cd({1: 1.0, 2: 1.20, 4: 1.18, 8: 1.195}) == 2
    assert pr.preferred_cd({1: 1.0, 2: 1.10, 4: 1.20, 8: 1.15}) == 4
    assert pr.preferred_cd({1: 1.0, 4: 2.126, 8: 2.111, 16: 1.925}) == 4
    assert pr.preferred_cd({1: 1.0, 2: 0.8, 16: 1.9}) == 16
    assert pr.preferred_cd({1: 1.0, 2: 1.3, 8: 1.3}) == 2            # exact tie: the smaller CD
    assert pr.preferred_cd({1: 1.0, 2: 0.9, 4: 0.7}) == 1            # concurrency only hurts
    assert pr.preferred_cd({1: 1.0}) == 1


def test_corun_rule_by_hand():
    # flags: bit 0 at once, bit 1 CD-2 kernel, bits 2-3 the op's cap index
    e_go = pr.Entry((7, 10, 12, 0), 4, (10, 11, 12, 13, 14), 0b0111)     # at once, CD-2 kernel, op GPU/2
    e_iso = pr.Entry((8, 10, 12, 0), 4, (30, 31, 32, 33, 34), 0b1001)    # at once, CD-1 kernel, op GPU/4
    e_off = pr.Entry((9, 10, 12, 0), 1, (20, 21, 22, 23, 24), 0)
    lut = pr.write_lut([e_go, e_iso, e_off], 132)
    d_go, d_iso, d_off = pr.Desc(128, 1024, 4096, 0), pr.Desc(256, 1024, 4096, 0), pr.Desc(512, 1024, 4096, 0)
    assert pr.corun_plan(d_go, lut, pr.POLICY_AUTO) == (1, 11, 2)
    assert pr.corun_plan(d_iso, lut, pr.POLICY_AUTO) == (1, 30, 4)
    assert pr.corun_plan(d_off, lut, pr.POLICY_AUTO) == (0, 20, 1)
    for d, e in ((d_go, e_go), (d_off, e_off)):
        assert pr.corun_plan(d, lut, pr.POLICY_SEQUENTIAL) == (0, e.variants[0], 1)
        assert pr.corun_plan(d, lut, pr.POLICY_DEFAULT) == (1, e.variants[0], 1)
        assert pr.corun_plan(d, lut, pr.POLICY_GO) == (1, e.variants[1], 2)
    with pytest.raises(pr.PlanError):
        pr.corun_plan(d_go, lut, pr.POLICY_FORCE_CD)
    # a batched GEMM is bucketed by M * batch rows
    assert pr.corun_plan(pr.Desc(64, 1024, 4096, 0, 2), lut, pr.POLICY_AUTO) == (1, 11, 2)


def test_lut_flag_bits_round_trip_and_validation():
    e = pr.Entry((7, 10, 12, 0), 4, (10, 11, 12, 13, 14), 0b1011)
    data = pr.write_lut([e], 132)
    assert data[32 + 5] == 0b1011
    assert pr.parse_lut(data)[0][0].flags == 0b1011
    for bad_flags in (0x10, 0b1100, 0x80):
        bad = bytearray(data)
        bad[32 + 5] = bad_flags
        with pytest.raises(pr.LutError):
            pr.parse_lut(bytes(bad))

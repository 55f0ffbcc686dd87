"""Reference restatement of the dynamic logic's table lookup —
TEST INFRASTRUCTURE ONLY.

The paper's dynamic logic inspects the pending independent GEMMs, predicts the
concurrency degree (CD) to run, and rewrites each GEMM's kernel to the
globally optimized kernel for that CD (Sec. 4.3, Sec. 4.4).  Here the
prediction is a lookup table profiled offline; this module restates, in plain
Python and independently of the product's C++ planner, how a schedule follows
from the table:

1. Bucket each GEMM by its sizes: key = (floor(log2 M), floor(log2 N),
   floor(log2 K), output dtype); a strided batch of GEMMs counts its rows
   over all entries (M * batch).  The paper's predictor reads M, N and K among
   its features (Sec. 4.3); a log2 bucket is this table's stand-in for them.
2. Look the key up.  A key the table lacks takes the stored key nearest in
   L1 distance over the three log2 sizes, a differing output dtype adding 16;
   ties go to the smallest stored key.  (Nearest-neighbour reuse of profiled
   GEMMs echoes the KNN tuning shortcut, Sec. 7.5.)
3. The CD actually run is the minimum of the preferred CD and the number of
   GEMMs available (Sec. 4.3).
4. Two or more distinct keys (heterogeneous GEMMs, Sec. 6.7): the paper runs
   the whole set at once only if every key prefers at least the set's size,
   and otherwise runs homogeneous groups, each with its own CD.  Generalized
   to any number of keys: one block per key, blocks in decreasing order of
   total FLOPs (ties: smaller key first), merged greedily with the next block
   while every key in the merged group still prefers at least the merged
   size.  With two keys this is exactly the paper's rule.  A single-key group
   runs at min(preferred CD, its size); a merged group runs all its members
   at once.
5. Inside a group GEMMs take stream slots round-robin (member j -> slot
   j mod CD), so at most CD run at once; each GEMM runs the table's kernel for
   the smallest CD class (1, 2, 4, 8, 16) not below the group's CD.
6. One kernel kind per wave (this build's rule for its fused launches, not
   the paper's): under the automatic policy, in each wave (a group's members
   taken CD at a time, in launch order) every GEMM other than the wave's
   largest (most FLOPs, ties: the first) takes the largest one's kernel kind,
   with no K split and the same grid-cap constraint, when that kind suits it:
   the same output dtype, K no longer than the largest one's, and M within
   the kind's reach (CTA-pair kind: M >= 128; transposed skinny-M kind:
   M <= 2 x its tile rows; other kinds: M >= 64).

Forced policies give the paper's comparison configurations through the same
schedule type (Sec. 5.5): ``sequential`` (isolation-tuned kernels one after
another), ``default`` (isolation-tuned kernels, all GEMMs at once on their own
streams), ``go`` (GO-Kernels, all GEMMs at once) and ``force_cd`` (GO-Kernels
at a fixed CD).

Binary formats written out here, independently of the C++ code:

LUT file (little-endian): 8-byte magic ``GOLDYLUT``, u32 version (1), u32
entry count, u32 variant-id bound, u32 SM count, 8 reserved bytes; then
16-byte entries ``u8 lm, u8 ln, u8 lk, u8 out_dtype, u8 pref_cd, u8 flags,
u16 variant[5]`` sorted strictly by (lm, ln, lk, out_dtype); flags record how
the bucket's GEMM runs with an element-wise op (bit 0 at once, bit 1 the CD-2
kernel, bits 2-3 the op's grid-cap divisor 1/2/4 as 0/1/2), other bits 0.

Schedule bytes (little-endian u32 words): ``GSCH`` magic, version (1),
n_gemms, n_groups, max_streams, flags; per group: cd, size, members...; per
GEMM: group, variant, slot.
"""
from __future__ import annotations

import struct
from dataclasses import dataclass
from typing import List, Optional, Sequence, Tuple

LUT_MAGIC = b"GOLDYLUT"
CD_CLASSES = (1, 2, 4, 8, 16)
MAX_GEMMS = 64
MAX_STREAMS = 16

# planning policies (low 4 bits of flags); the forced CD sits in bits 8..15
POLICY_AUTO = 0
POLICY_SEQUENTIAL = 1
POLICY_DEFAULT = 2
POLICY_GO = 3
POLICY_FORCE_CD = 4
FUSED = 0x10            # launch-mode bit: does not change the plan, only how it is launched

DTYPE_BF16 = 0
DTYPE_F32 = 1


class LutError(ValueError):
    pass


class PlanError(ValueError):
    pass


@dataclass(frozen=True)
class Entry:
    key: Tuple[int, int, int, int]
    pref_cd: int
    variants: Tuple[int, int, int, int, int]
    flags: int = 0          # co-run with an element-wise op: bit 0 at once, bit 1 CD-2 kernel, bits 2-3 op cap


def parse_lut(data: bytes) -> Tuple[List[Entry], int]:
    """Entries and the variant-id bound of a LUT file; raises LutError on any
    malformed field."""
    if len(data) < 32 or data[:8] != LUT_MAGIC:
        raise LutError("bad magic")
    version, n, n_variants, _sm = struct.unpack_from("<IIII", data, 8)
    if version != 1:
        raise LutError("bad version")
    if len(data) != 32 + 16 * n:
        raise LutError("bad size")
    entries: List[Entry] = []
    prev = None
    for e in range(n):
        lm, ln, lk, out, pref, flags = struct.unpack_from("<6B", data, 32 + 16 * e)
        vs = struct.unpack_from("<5H", data, 32 + 16 * e + 6)
        key = (lm, ln, lk, out)
        if prev is not None and key <= prev:
            raise LutError("entries not strictly sorted")
        if out not in (DTYPE_BF16, DTYPE_F32):
            raise LutError("bad dtype")
        if pref not in CD_CLASSES:
            raise LutError("bad preferred cd")
        if flags & ~0x0F or (flags >> 2) & 3 == 3:
            raise LutError("unknown flag bits")
        if any(v >= n_variants for v in vs):
            raise LutError("variant out of range")
        prev = key
        entries.append(Entry(key, pref, tuple(vs), flags))
    if not entries:
        raise LutError("empty table")
    return entries, n_variants


def write_lut(entries: Sequence[Entry], n_variants: int, sm_count: int = 0) -> bytes:
    out = bytearray(LUT_MAGIC)
    out += struct.pack("<IIIIII", 1, len(entries), n_variants, sm_count, 0, 0)
    for e in sorted(entries, key=lambda x: x.key):
        out += struct.pack("<6B", *e.key, e.pref_cd, e.flags)
        out += struct.pack("<5H", *e.variants)
    return bytes(out)


def floor_log2(x: int) -> int:
    """floor(log2 x) for x >= 1, and 0 for x == 0, clamped to a byte."""
    if x <= 0:
        return 0
    return min(x.bit_length() - 1, 255)


def bucket_key(M: int, N: int, K: int, out_dtype: int) -> Tuple[int, int, int, int]:
    return (floor_log2(M), floor_log2(N), floor_log2(K), out_dtype)


def lookup(entries: Sequence[Entry], key) -> Entry:
    best = None
    best_d = None
    for e in entries:                       # entries are in increasing key order
        d = (abs(e.key[0] - key[0]) + abs(e.key[1] - key[1]) + abs(e.key[2] - key[2])
             + (16 if e.key[3] != key[3] else 0))
        if best_d is None or d < best_d:    # strict: earlier (smaller) key wins ties
            best, best_d = e, d
    return best


# Kernel kinds of the variant registry, written out from the library's
# documented layout (variant id = (kind * 4 + split index) * 3 + grid-cap
# index): kind -> (tensor-core tile columns, transposed skinny-M tile, CTA
# pair).  Transposed kinds cover mma_n rows of C per tile.
KINDS = {
    0: (64, False, False), 1: (64, False, False), 2: (128, False, False), 3: (128, False, False),
    4: (256, False, False), 5: (256, False, False), 6: (32, True, False), 7: (32, True, False),
    8: (64, True, False), 9: (64, True, False), 10: (256, False, True),
}


def kind_of(variant: int) -> int:
    return variant // 12


def same_kind_variant(kind: int, like_variant: int) -> int:
    """Variant of `kind` with no K split and the grid-cap index of `like_variant`."""
    return (kind * 4 + 0) * 3 + like_variant % 3


def kind_suits(kind: int, M: int) -> bool:
    mma_n, swap, pair = KINDS[kind]
    if pair:
        return M >= 128
    if swap:
        return M <= 2 * mma_n
    return M >= 64


def one_kind_per_wave(descs: Sequence["Desc"], groups):
    """Rule 6 over groups given as (cd, members, variants); returns new groups."""
    out = []
    for cd, members, variants in groups:
        var = dict(zip(members, variants))
        for w0 in range(0, len(members), max(1, cd)):
            wave = members[w0:w0 + max(1, cd)]
            flops = [2 * descs[i].M * descs[i].N * descs[i].K * descs[i].batch for i in wave]
            dom = wave[flops.index(max(flops))]            # the first of the largest
            kd = kind_of(var[dom])
            for i in wave:
                if i == dom or kind_of(var[i]) == kd:
                    continue
                if descs[i].out_dtype != descs[dom].out_dtype or descs[i].K > descs[dom].K:
                    continue
                if kind_suits(kd, descs[i].M):
                    var[i] = same_kind_variant(kd, var[dom])
        out.append((cd, members, [var[i] for i in members]))
    return out


def cd_class_index(cd: int) -> int:
    for idx, c in enumerate(CD_CLASSES):
        if cd <= c:
            return idx
    return len(CD_CLASSES) - 1


@dataclass(frozen=True)
class Desc:
    M: int
    N: int
    K: int
    out_dtype: int
    batch: int = 1          # strided batch entries (Sec. 6.7's B-GEMMs); bucketed by M * batch rows


def plan(descs: Sequence[Desc], lut_bytes: bytes, flags: int = 0):
    """Schedule as (groups, per_gemm, max_streams, flags): groups is a list of
    (cd, members); per_gemm[i] = (group, variant, slot)."""
    entries, _ = parse_lut(lut_bytes)
    n = len(descs)
    if n < 1 or n > MAX_GEMMS:
        raise PlanError("bad count")
    policy = flags & 0xF
    forced = (flags >> 8) & 0xFF
    if (flags & ~0xFF1F) or policy > POLICY_FORCE_CD or (policy == POLICY_FORCE_CD and forced < 1):
        raise PlanError("bad flags")
    keys = [bucket_key(d.M * d.batch, d.N, d.K, d.out_dtype) for d in descs]
    ents = [lookup(entries, k) for k in keys]

    def one_group(cd: int, cls_cd: Optional[int]):
        cd = max(1, min(cd, n, MAX_STREAMS))
        ci = cd_class_index(cd if cls_cd is None else cls_cd)
        members = list(range(n))
        return [(cd, members, [ents[i].variants[ci] for i in members])]

    if policy == POLICY_SEQUENTIAL:
        groups = one_group(1, 1)
    elif policy == POLICY_DEFAULT:
        groups = one_group(n, 1)
    elif policy == POLICY_GO:
        groups = one_group(n, None)
    elif policy == POLICY_FORCE_CD:
        groups = one_group(forced, None)
    else:
        blocks = []
        for k in sorted(set(keys)):
            members = [i for i in range(n) if keys[i] == k]
            flops = sum(2 * descs[i].M * descs[i].N * descs[i].K * descs[i].batch for i in members)
            blocks.append((-flops, k, members, ents[members[0]].pref_cd))
        blocks.sort(key=lambda b: (b[0], b[1]))
        merged = []                         # each: (members, min pref, n keys)
        for _, _, members, pref in blocks:
            if merged:
                cur_members, cur_pref, cur_keys = merged[-1]
                size = len(cur_members) + len(members)
                if min(cur_pref, pref) >= size:
                    merged[-1] = (cur_members + members, min(cur_pref, pref), cur_keys + 1)
                    continue
            merged.append((list(members), pref, 1))
        groups = []
        for members, pref, n_keys in merged:
            cd = len(members) if n_keys > 1 else min(pref, len(members))
            cd = max(1, min(cd, MAX_STREAMS))
            ci = cd_class_index(cd)
            groups.append((cd, members, [ents[i].variants[ci] for i in members]))
        groups = one_kind_per_wave(descs, groups)

    per_gemm = [None] * n
    for g, (cd, members, variants) in enumerate(groups):
        for j, (i, v) in enumerate(zip(members, variants)):
            per_gemm[i] = (g, v, j % cd)
    max_streams = max(cd for cd, _, _ in groups)
    return [(cd, members) for cd, members, _ in groups], per_gemm, max_streams, flags


def serialize(schedule) -> bytes:
    groups, per_gemm, max_streams, flags = schedule
    words = [0x48435347, 1, len(per_gemm), len(groups), max_streams, flags & 0xFFFFFFFF]
    for cd, members in groups:
        words += [cd, len(members)] + list(members)
    for g, v, s in per_gemm:
        words += [g, v, s]
    return struct.pack("<%dI" % len(words), *words)


def preferred_cd(speedup: dict, gain: float = 0.05) -> int:
    """Preferred CD from measured speedups over serial execution.

    Sec. 4.3 (Dynamic logic for concurrency control): a GEMM's preferred CD
    is the CD under which it shows the most speedup.  Sec. 5.5
    (Configurations): the paper's Oracle runs the GEMMs sequentially unless
    some CD gains at least 5% over sequential.  So: the largest speedup among
    the CD classes wins; exact ties go to the smaller CD (the paper does not
    address ties; the smaller CD shares the GPU among fewer GEMMs); CD 1
    unless that largest speedup reaches 1 + ``gain``.  ``speedup[1]`` is 1
    by definition."""
    best_cd, best = 1, 1.0
    for cd in CD_CLASSES[1:]:
        if cd in speedup and speedup[cd] > best:
            best_cd, best = cd, speedup[cd]
    return best_cd if best >= 1.0 + gain else 1


def corun_plan(d: Desc, lut_bytes: bytes, policy: int) -> Tuple[int, int, int]:
    """A GEMM co-scheduled with an element-wise op over its output (Sec. 7.1):
    (concurrent, GEMM variant, grid-cap divisor of the element-wise kernel).
    sequential: isolation-tuned kernel, then the op; default: the
    isolation-tuned kernel and the op (whole GPU) at once; go: the CD-2
    GO-Kernel and the op capped at half the GPU, at once; automatic: the
    configuration the table entry's flags record (bit 0 at once, bit 1 the
    CD-2 kernel instead of the CD-1 one, bits 2-3 the op's cap 1, 2 or 4),
    one after the other when bit 0 is clear — concurrency restricted where it
    does not help."""
    entries, _ = parse_lut(lut_bytes)
    if policy not in (POLICY_AUTO, POLICY_SEQUENTIAL, POLICY_DEFAULT, POLICY_GO):
        raise PlanError("bad policy")
    e = lookup(entries, bucket_key(d.M * d.batch, d.N, d.K, d.out_dtype))
    if policy == POLICY_SEQUENTIAL:
        return 0, e.variants[0], 1
    if policy == POLICY_DEFAULT:
        return 1, e.variants[0], 1
    if policy == POLICY_GO:
        return 1, e.variants[1], 2
    if e.flags & 1:
        return 1, e.variants[1] if e.flags & 2 else e.variants[0], 1 << ((e.flags >> 2) & 3)
    return 0, e.variants[0], 1

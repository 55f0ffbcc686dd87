"""Reference restatement of the logistic-regression CD predictor —
TEST INFRASTRUCTURE ONLY.

The paper trains, once per GPU, a multi-class logistic regression that maps a
GEMM to its preferred concurrency degree (Sec. 4.3, Eq. 1).  This module
restates, in plain Python and independently of the product's C++ planner,
what the trained model computes at planning time:

1. Features (Sec. 4.3): the GEMM's M (times its batch), N and K, and for each CD class c in
   (1, 2, 4, 8, 16) three numbers of the GO-Kernel the table assigns to the
   GEMM's bucket at that CD — its work-group count (here: CTAs of work, i.e.
   output tiles x split-K slices, two CTAs per tile for a CTA-pair kernel),
   its occupancy (CTAs resident per SM) and its wave count (CTAs of work over
   the CTAs its capped persistent grid keeps resident, rounded up).  Eighteen
   features in that order.
2. Min-max normalisation with the training set's per-feature minimum and
   maximum: (x - lo) / (hi - lo), 0 where hi == lo.
3. Scores s_c = b_c + sum_j W[c][j] x_j (j in increasing order), and Eq. 1's
   probabilities P_c = exp(s_c) / sum_i exp(s_i).  The prediction is the CD
   class of largest probability — equivalently of largest score, since exp is
   increasing; ties go to the smaller CD.
4. The CD run is min(prediction, GEMMs available) (Sec. 4.3); with several
   GEMMs of one bucket the planner takes the smallest of their predictions.

Model file (little-endian): 8-byte magic ``GOLDYLRM``, u32 version (1), u32
feature count (18), u32 class count (5), u32 SM count, 8 reserved bytes; then
f64 lo[18], f64 hi[18], f64 W[5][18] (class-major), f64 b[5].

GO-Kernel geometry needed for the features, written out here from the kernel
design (kind = variant // 12, split = (1, 2, 4, 8)[(variant // 3) % 4], grid
cap divisor = (1, 2, 4)[variant % 3]):

  kind  tile (rows x cols of C)  CTAs/SM  CTAs per tile
  0     128 x 64                 1        1
  1     128 x 64                 2        1
  2     128 x 128                1        1
  3     128 x 128                2        1
  4     128 x 256                1        1
  5     128 x 256                2        1
  6     32 x 128                 1        1
  7     32 x 128                 2        1
  8     64 x 128                 1        1
  9     64 x 128                 2        1
  10    256 x 256                1        2   (split-K never used)
"""
from __future__ import annotations

import math
import struct
from dataclasses import dataclass
from typing import List, Optional, Sequence, Tuple

from . import planner_ref as pr

MAGIC = b"GOLDYLRM"
N_FEATURES = 18
N_CLASSES = 5

# kind -> (tile rows, tile cols, CTAs per SM, CTAs per tile)
KIND_GEOMETRY = {
    0: (128, 64, 1, 1), 1: (128, 64, 2, 1),
    2: (128, 128, 1, 1), 3: (128, 128, 2, 1),
    4: (128, 256, 1, 1), 5: (128, 256, 2, 1),
    6: (32, 128, 1, 1), 7: (32, 128, 2, 1),
    8: (64, 128, 1, 1), 9: (64, 128, 2, 1),
    10: (256, 256, 1, 2),
}
SPLITS = (1, 2, 4, 8)
RC_DIVS = (1, 2, 4)


class ModelError(ValueError):
    pass


@dataclass(frozen=True)
class Model:
    lo: Tuple[float, ...]
    hi: Tuple[float, ...]
    W: Tuple[Tuple[float, ...], ...]
    b: Tuple[float, ...]
    sm_count: int


def parse_model(data: bytes) -> Model:
    if len(data) < 32 or data[:8] != MAGIC:
        raise ModelError("bad magic")
    version, nf, nc, sm = struct.unpack_from("<IIII", data, 8)
    if version != 1 or nf != N_FEATURES or nc != N_CLASSES:
        raise ModelError("bad version or shape")
    if sm == 0:
        raise ModelError("sm count is zero")
    if len(data) != 32 + 8 * (2 * nf + nc * nf + nc):
        raise ModelError("bad size")
    vals = struct.unpack_from("<%dd" % (2 * nf + nc * nf + nc), data, 32)
    if not all(math.isfinite(v) for v in vals):
        raise ModelError("non-finite value")
    lo = vals[:nf]
    hi = vals[nf:2 * nf]
    if any(h < l for l, h in zip(lo, hi)):
        raise ModelError("hi below lo")
    W = tuple(tuple(vals[2 * nf + c * nf: 2 * nf + (c + 1) * nf]) for c in range(nc))
    b = tuple(vals[2 * nf + nc * nf:])
    return Model(tuple(lo), tuple(hi), W, b, sm)


def write_model(m: Model) -> bytes:
    out = bytearray(MAGIC)
    out += struct.pack("<IIIIII", 1, N_FEATURES, N_CLASSES, m.sm_count, 0, 0)
    vals = list(m.lo) + list(m.hi) + [w for row in m.W for w in row] + list(m.b)
    out += struct.pack("<%dd" % len(vals), *vals)
    return bytes(out)


def kernel_features(M: int, N: int, variant: int, sm_count: int, batch: int = 1) -> Tuple[int, int, int]:
    """(CTAs of work, CTAs per SM, waves) of one GO-Kernel on `batch` M x N
    outputs."""
    kind = variant // 12
    split = SPLITS[(variant // 3) % 4]
    rc_div = RC_DIVS[variant % 3]
    rows, cols, per_sm, per_tile = KIND_GEOMETRY[kind]
    tiles = batch * (-(-M // rows)) * (-(-N // cols))
    ctas = tiles * split * per_tile
    cap = max(per_tile, per_sm * sm_count // rc_div)
    waves = -(-ctas // cap)
    return ctas, per_sm, waves


def features(d: pr.Desc, entry: pr.Entry, sm_count: int) -> List[float]:
    x = [float(d.M * d.batch), float(d.N), float(d.K)]
    for v in entry.variants:
        x += [float(f) for f in kernel_features(d.M, d.N, v, sm_count, d.batch)]
    return x


def normalise(x: Sequence[float], m: Model) -> List[float]:
    return [(xi - l) / (h - l) if h > l else 0.0 for xi, l, h in zip(x, m.lo, m.hi)]


def scores(xn: Sequence[float], m: Model) -> List[float]:
    out = []
    for c in range(N_CLASSES):
        s = m.b[c]
        for j in range(N_FEATURES):
            s = s + m.W[c][j] * xn[j]
        out.append(s)
    return out


def probabilities(s: Sequence[float]) -> List[float]:
    """Eq. 1: softmax over the class scores."""
    top = max(s)
    e = [math.exp(v - top) for v in s]
    tot = sum(e)
    return [v / tot for v in e]


def predict_class(s: Sequence[float]) -> int:
    best = 0
    for c in range(1, N_CLASSES):
        if s[c] > s[best]:
            best = c
    return best


def predict_cd(d: pr.Desc, entries: Sequence[pr.Entry], m: Model) -> int:
    e = pr.lookup(entries, pr.bucket_key(d.M * d.batch, d.N, d.K, d.out_dtype))
    s = scores(normalise(features(d, e, m.sm_count), m), m)
    return pr.CD_CLASSES[predict_class(s)]


def plan(descs: Sequence[pr.Desc], lut_bytes: bytes, model_bytes: Optional[bytes], flags: int = 0):
    """The planner with the predictor supplying each bucket's preferred CD
    (the smallest prediction over the bucket's GEMMs) under the automatic
    policy; the forced policies and a missing model plan as planner_ref."""
    if model_bytes is None or (flags & 0xF) != pr.POLICY_AUTO:
        return pr.plan(descs, lut_bytes, flags)
    m = parse_model(model_bytes)
    entries, _ = pr.parse_lut(lut_bytes)
    prefs = {}
    for d in descs:
        k = pr.bucket_key(d.M * d.batch, d.N, d.K, d.out_dtype)
        prefs[k] = min(prefs.get(k, pr.CD_CLASSES[-1]), predict_cd(d, entries, m))
    return _plan_with_prefs(descs, entries, prefs, flags)


def _plan_with_prefs(descs, entries, prefs, flags):
    n = len(descs)
    if n < 1 or n > pr.MAX_GEMMS:
        raise pr.PlanError("bad count")
    if flags & ~0xFF1F:
        raise pr.PlanError("bad flags")
    keys = [pr.bucket_key(d.M * d.batch, d.N, d.K, d.out_dtype) for d in descs]
    ents = [pr.lookup(entries, k) for k in keys]
    blocks = []
    for k in sorted(set(keys)):
        members = [i for i in range(n) if keys[i] == k]
        flops = sum(2 * descs[i].M * descs[i].N * descs[i].K * descs[i].batch for i in members)
        blocks.append((-flops, k, members, prefs[k]))
    blocks.sort(key=lambda b: (b[0], b[1]))
    merged = []
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
        cd = max(1, min(cd, pr.MAX_STREAMS))
        ci = pr.cd_class_index(cd)
        groups.append((cd, members, [ents[i].variants[ci] for i in members]))
    groups = pr.one_kind_per_wave(descs, groups)
    per_gemm = [None] * n
    for g, (cd, members, variants) in enumerate(groups):
        for j, (i, v) in enumerate(zip(members, variants)):
            per_gemm[i] = (g, v, j % cd)
    max_streams = max(cd for cd, _, _ in groups)
    return [(cd, members) for cd, members, _ in groups], per_gemm, max_streams, flags

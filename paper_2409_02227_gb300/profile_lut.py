"""Offline profiler that builds the dynamic logic's lookup table on the GPU.

It follows the paper's one-time tuning (Sec. 4.2.1, Sec. 4.3) per shape
bucket, with this build's GO-Kernel variants standing in for Tensile's kernel
list:

  step 1 (resource-constrained tuning): time every candidate kernel (tile
         kind x split-K) alone under three resource constraints — persistent
         grid capped at the whole GPU, half and a quarter of it (the paper's
         GPU, GPU/2, GPU/4; shared L2 cannot be partitioned here, so
         contention for it is only seen in step 2) — and keep the fastest per
         constraint;
  step 2 (concurrent benchmarking): for each concurrency degree CD in
         {2, 4, 8, 16}, co-run CD copies of the GEMM (distinct buffers) with
         each step-1 winner, launched the way the library will launch them
         (one fused launch by default, or one stream each); the fastest is
         the GO-Kernel for that CD.  The CD-1 kernel is the whole-GPU winner (the
         isolation-tuned kernel);
  preferred CD: speedup(CD) = CD * T(1) / T(CD) over running the copies one
         after another; the largest wins (exact ties: the smaller CD), but
         sequential (CD 1) unless some CD gains at least 5% (Sec. 5.5).

Each bucket (floor log2 of M, N, K; output dtype) is profiled at two
points: its lower edge (M, N, K = powers of two), where DNN layer sizes
usually sit, and its geometric centre (2^(l + 1/2), N and K rounded to 64).
A candidate's score is its mean time relative to the fastest candidate at
each point, and speedups are averaged over the points, so that a choice holds
across the bucket (a table profiled at the lower edges alone ran the
randomized sets, whose shapes fill the buckets, 7% slower).  Timing:
prepared runs (recorded plain launches, the way the benchmark replays a step)
back to back on one stream, as the paper ran GEMMs back to back on each
stream (Sec. 5.3), rotating over disjoint copies of the operands so that they
come from HBM as in the benchmark (inputs rotated past twice the L2); the
median of several repetitions of a timed batch.  Runs are recorded without
inputs_ready, so that one replay does not overlap the next: a co-run's time
is the makespan of its CD GEMMs, as the paper measures it (with overlapping
replays, kernels whose small grids let consecutive co-runs run side by side
win, and the table then chose worse kernels for heterogeneous waves, whose
launches do not overlap across steps: randomized sets 0.358 -> 0.349 of
roofline, hetero_pair 45.8 -> 52.8 us); ``--inputs-ready`` profiles with it.
Results are appended to a JSONL log bucket by bucket, so an interrupted run
resumes where it stopped; the LUT file is written at the end.

With ``--dataset FILE`` it instead records the CD predictor's training set
(Sec. 4.3): for each of the dataset GEMMs, the co-run time at every CD class
with the table's GO-Kernel for that CD.

Usage (on a GPU):  python -m paper_2409_02227_gb300.profile_lut --out DIR
                   [--configs] [--sweep] [--keys lm,ln,lk,out ...]
                   python -m paper_2409_02227_gb300.profile_lut --dataset FILE
"""
from __future__ import annotations

import argparse
import json
import math
import os
import struct
import sys
import time
from typing import Dict, List, Sequence, Tuple

import torch

from . import goldy as G
from . import workloads as wl

CD_CLASSES = (1, 2, 4, 8, 16)
RC_DIVS = (1, 2, 4)
SPLITS = (1, 2, 4, 8)
SWAP_KINDS = (6, 7, 8, 9)
NONSWAP_KINDS = (0, 1, 2, 3, 4, 5)
PAIR_KINDS = (10,)


def write_lut(entries, n_variants: int, sm_count: int) -> bytes:
    """LUT bytes in the format goldy_lut_load reads (include/goldy.h) from
    (key, preferred CD, variants[, flags]) tuples."""
    out = bytearray(b"GOLDYLUT")
    out += struct.pack("<IIIIII", 1, len(entries), n_variants, sm_count, 0, 0)
    for e in sorted(entries, key=lambda e: e[0]):
        key, pref, variants = e[0], e[1], e[2]
        flags = e[3] if len(e) > 3 else 0
        out += bytes([key[0], key[1], key[2], key[3], pref, flags])
        out += struct.pack("<5H", *variants)
    return bytes(out)


def preferred_cd(speedup: Dict[int, float], gain: float = 0.05) -> int:
    """The CD with the largest speedup over running the copies one after
    another (Sec. 4.3), exact ties to the smaller CD; sequential (1) unless
    that speedup reaches 1 + ``gain`` (Sec. 5.5's Oracle configuration)."""
    best_cd, best = 1, 1.0
    for cd in (2, 4, 8, 16):
        if cd in speedup and speedup[cd] > best:
            best_cd, best = cd, speedup[cd]
    return best_cd if best >= 1.0 + gain else 1


def logged_pref(rec: dict) -> int:
    """Preferred CD of a logged bucket under the current rule."""
    return preferred_cd({int(c): v for c, v in rec["speedup"].items()})


def bucket_shape(key) -> Tuple[int, int, int, int]:
    lm, ln, lk, out = key
    return 1 << lm, max(64, 1 << ln), max(64, 1 << lk), out


def bucket_centre(key) -> Tuple[int, int, int, int]:
    """Geometric centre of a bucket: 2^(l + 1/2) per size, N and K rounded to
    multiples of 64 (as the workloads' N and K are)."""
    lm, ln, lk, out = key
    c = lambda l: 2.0 ** (l + 0.5)
    return (max(1, int(round(c(lm)))), max(64, 64 * int(round(c(ln) / 64))), max(64, 64 * int(round(c(lk) / 64))),
            out)


def bucket_points(key) -> List[Tuple[int, int, int, int]]:
    """Sample points a bucket is profiled at: its lower edge and its centre."""
    pts = [bucket_shape(key)]
    if bucket_centre(key) != pts[0]:
        pts.append(bucket_centre(key))
    return pts


def candidates(M: int, N: int, K: int, sm_count: int) -> List[Tuple[int, int]]:
    kinds = (list(NONSWAP_KINDS) + (list(SWAP_KINDS) if M <= 128 else [])
             + (list(PAIR_KINDS) if M > 128 else []))
    k_blocks = math.ceil(K / 64)
    out = []
    for kind in kinds:
        info = G.goldy_variant_info_get(G.variant_id(kind, 1, 1))
        rows = info["mma_n"] if info["swap_ab"] else info["mma_m"]
        cols = 128 if info["swap_ab"] else info["mma_n"]
        tiles = math.ceil(M / rows) * math.ceil(N / cols)
        for s in SPLITS:
            if s > 1 and (s > k_blocks or tiles * s > 4 * sm_count):
                continue
            out.append((kind, s))
    return out


class Bench:
    """Device copies of one GEMM, timed as prepared runs replayed back to back
    on the bench's streams (or a partition's).  A co-run of c copies is
    prepared once per disjoint group of c copies and the replays rotate over
    the groups, so that — as in the benchmark — the inputs touched between
    two uses of the same copy exceed twice the L2 and every GEMM reads its
    operands from HBM."""

    def __init__(self, M: int, N: int, K: int, out: int, copies: int = 16, seed: int = 0, partition=None,
                 rotate: bool = True, max_bytes: int = 6 << 30, inputs_ready: bool = False):
        self.M, self.N, self.K, self.out = M, N, K, out
        self.partition = partition
        self.inputs_ready = inputs_ready
        cdt = torch.float32 if out == G.GOLDY_F32 else torch.bfloat16
        per = 2 * M * K + 2 * K * N
        cbytes = M * N * (4 if out == G.GOLDY_F32 else 2)
        l2 = int(getattr(torch.cuda.get_device_properties(torch.cuda.current_device()), "L2_cache_size", 126 << 20))
        total = copies
        if rotate:
            total = max(copies, -(-2 * l2 // max(per, 1)) + copies)
            total = min(total, max(copies, max_bytes // max(per + cbytes, 1)))
        self.total = total
        gen = torch.Generator(device="cuda")
        gen.manual_seed(seed)
        self.A = [(torch.rand((M, K), generator=gen, device="cuda") - 0.5).to(torch.bfloat16) for _ in range(total)]
        self.B = [(torch.rand((K, N), generator=gen, device="cuda") - 0.5).to(torch.bfloat16) for _ in range(total)]
        self.C = [torch.empty((M, N), dtype=cdt, device="cuda") for _ in range(total)]
        self.streams = [torch.cuda.Stream() for _ in range(16)]
        self.part_streams = (G.goldy_partition_query(partition, 16)[1] if partition is not None
                             else [st.cuda_stream for st in self.streams])
        self.ws = None

    def _workspace(self, nbytes: int) -> torch.Tensor:
        if self.ws is None or self.ws.numel() < nbytes:
            self.ws = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device="cuda")
        return self.ws

    def time_us(self, variant: int, copies: int, concurrent: bool, target_us: float = 2000.0,
                fused: bool = True, samples: int = 5) -> float:
        """Median time of one co-run of `copies` GEMMs with `variant` (samples
        = 0: quick mode, a single replay when it alone reaches target_us)."""
        d = G.desc(self.M, self.N, self.K, self.out)
        slots = list(range(copies)) if concurrent else [0] * copies
        sched = G.goldy_schedule_build([d] * copies, [0] * copies, [variant] * copies, slots,
                                       G.GOLDY_PLAN_FUSED if fused else 0)
        _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
        ws = self._workspace(ws_bytes)
        torch.cuda.synchronize()
        groups = max(1, self.total // copies)
        execs = []
        for r in range(groups):
            lo, hi = r * copies, (r + 1) * copies
            execs.append(G.goldy_exec_create(sched, [a.data_ptr() for a in self.A[lo:hi]],
                                             [b.data_ptr() for b in self.B[lo:hi]],
                                             [c.data_ptr() for c in self.C[lo:hi]], ws.data_ptr(), ws_bytes,
                                             self.part_streams[:max(1, ms)], inputs_ready=self.inputs_ready))
        est = max(G.goldy_exec_time(execs, min(groups, 3 if samples else 1), 1) * 1e3, 1.0)
        if samples == 0:
            if est >= target_us:
                del execs
                return est
            samples = 3
        reps = int(min(2000, max(3, target_us / est)))
        times = sorted(G.goldy_exec_time(execs, 0, reps) * 1e3 for _ in range(samples))
        del execs
        if G.goldy_device_error(clear=True) != 0:
            raise RuntimeError("kernel reported a bounded-wait timeout while profiling")
        return times[len(times) // 2]


def rank_variants(times: Dict[int, Sequence[float]]) -> List[int]:
    """Variants from best to worst by the mean, over the sample points, of
    their time relative to the fastest variant at that point (ties: the
    smaller id)."""
    n = len(next(iter(times.values())))
    fastest = [min(ts[pi] for ts in times.values()) for pi in range(n)]
    score = {v: sum(t / f for t, f in zip(ts, fastest)) / n for v, ts in times.items()}
    return sorted(times, key=lambda v: (score[v], v))


def pick_variant(times: Dict[int, Sequence[float]]) -> int:
    """The best variant of rank_variants."""
    return rank_variants(times)[0]


def profile_bucket(key, sm_count: int, log, fused: bool = True, partition=None, inputs_ready: bool = False,
                   top: int = 1) -> dict:
    """Steps 1 and 2 for one bucket, at each of its sample points; a variant's
    score is its mean time relative to the fastest candidate at each point,
    so that the choice holds across the bucket, not at one shape only."""
    points = bucket_points(key)
    M, N, K, out = points[0]
    benches = [Bench(*pt, partition=partition, inputs_ready=inputs_ready) for pt in points]
    cands = sorted(set().union(*[set(candidates(pt[0], pt[1], pt[2], sm_count)) for pt in points]))
    rows = []

    def ranked(variants, copies, step, extra):
        times = {v: [b.time_us(v, copies, True, fused=fused) for b in benches] for v in variants}
        for v, ts in times.items():
            for pi, t in enumerate(ts):
                rows.append(dict(step=step, variant=v, point=pi, us=t, **extra))
        order = rank_variants(times)
        return order, times

    winners = {}
    for rc in RC_DIVS:                                  # step 1
        winners[rc] = ranked([G.variant_id(kind, split, rc) for kind, split in cands], 1, 1, {"rc": rc})
    go = {1: winners[1][0][0]}
    t_cd = {1: winners[1][1][go[1]]}
    # step 2 co-runs the best `top` kernels of each constraint (the paper: the best one)
    step2 = sorted({v for rc in RC_DIVS for v in winners[rc][0][:top]})
    for cd in (2, 4, 8, 16):                            # step 2
        order, times = ranked(step2, cd, 2, {"cd": cd})
        go[cd], t_cd[cd] = order[0], times[order[0]]
    # speedup over running the copies one after another, averaged over the points
    speedup = {cd: sum(cd * t1 / tc for t1, tc in zip(t_cd[1], t_cd[cd])) / len(points) for cd in CD_CLASSES}
    pref = preferred_cd(speedup)
    rec = {"key": list(key), "shape": [M, N, K, out], "points": [list(pt) for pt in points], "pref_cd": pref,
           "launch": "fused" if fused else "streams", "inputs_ready": bool(inputs_ready),
           "variants": [go[c] for c in CD_CLASSES],
           "t_us": {str(c): t_cd[c][0] for c in CD_CLASSES},
           "t_us_points": {str(c): t_cd[c] for c in CD_CLASSES},
           "speedup": {str(c): speedup[c] for c in CD_CLASSES}, "rows": rows}
    log.write(json.dumps(rec) + "\n")
    log.flush()
    del benches
    torch.cuda.empty_cache()
    return rec





CORUN_CONFIGS = [(f"v{vi}_rc{1 << ri}", 1 | (vi << 1) | (ri << 2)) for vi in (0, 1) for ri in (0, 1, 2)]


def corun_times(bench: "Bench", variants: Sequence[int], target_us: float = 2000.0) -> Dict[str, float]:
    """Step 3 (Sec. 7.1): the bucket's GEMM with an element-wise add of its
    output size, one after the other ("sequential": the CD-1 kernel, then the
    add over the whole GPU) and at once in every configuration the table can
    record: the CD-1 or the CD-2 GO-Kernel ("v0", "v1") with the add's grid
    capped at GPU, GPU/2 or GPU/4 ("rc1", "rc2", "rc4").  Rotates over the
    bench's copies like time_us."""
    M, N, K, out = bench.M, bench.N, bench.K, bench.out
    n = M * N
    cdt = torch.float32 if out == G.GOLDY_F32 else torch.bfloat16
    R = max(1, bench.total // 2)              # the add's operands double the bytes per copy
    if getattr(bench, "X", None) is None:
        bench.X = [torch.randn(n, device="cuda").to(cdt) for _ in range(R)]
        bench.Y = [torch.randn(n, device="cuda").to(cdt) for _ in range(R)]
        bench.Z = [torch.empty(n, device="cuda", dtype=cdt) for _ in range(R)]
    streams = bench.part_streams[:2]
    t = {}
    for name, flags in [("sequential", 0)] + CORUN_CONFIGS:
        lut = G.goldy_lut_from_memory(write_lut([((0, 0, 0, out), 2, list(variants), flags)],
                                                G.goldy_variant_count(), 0))
        c = G.goldy_corun_plan(G.desc(M, N, K, out), n, out, lut, G.GOLDY_PLAN_AUTO)
        _, _, _, ws_bytes = G.goldy_corun_query(c)
        ws = bench._workspace(ws_bytes)
        torch.cuda.synchronize()
        execs = [G.goldy_corun_exec_create(c, bench.A[r].data_ptr(), bench.B[r].data_ptr(), bench.C[r].data_ptr(),
                                           ws.data_ptr(), ws_bytes, bench.X[r].data_ptr(), bench.Y[r].data_ptr(),
                                           bench.Z[r].data_ptr(), streams) for r in range(R)]
        est = max(G.goldy_exec_time(execs, min(R, 3), 1) * 1e3, 1.0)
        reps = int(min(2000, max(3, target_us / est)))
        t[name] = sorted(G.goldy_exec_time(execs, 0, reps) * 1e3 for _ in range(5))[2]
        del execs
    if G.goldy_device_error(clear=True) != 0:
        raise RuntimeError("kernel reported a bounded-wait timeout while profiling")
    return t


def corun_flags(t: Dict[str, float], gain: float = 0.05) -> int:
    """The table's co-run flags from step 3's times, with the preferred-CD
    rule's 5% threshold (Sec. 5.5) applied twice: a configuration other than
    the default one (CD-1 kernel, add over the whole GPU) is recorded only
    when it beats the default by `gain`, and running at once at all only when
    the chosen configuration beats one after the other by `gain` (0:
    sequential).  Small differences between profiled configurations do not
    carry over from a bucket's sample shape to the rest of the bucket."""
    default = "v0_rc1"
    name, flags = min(CORUN_CONFIGS, key=lambda c: (t[c[0]], c[1]))
    if t[name] * (1.0 + gain) > t[default]:
        name, flags = default, 1
    return flags if t[name] * (1.0 + gain) <= t["sequential"] else 0


def add_corun_flags(out_dir: str, fused: bool, partition=None) -> None:
    """Step 3 over a profiled table: time every bucket's GEMM + element-wise
    add in each configuration and record the chosen one in the entry's flags."""
    prof = os.path.join(out_dir, "profile.jsonl")
    recs = {}
    for line in open(prof):
        r = json.loads(line)
        recs[tuple(r["key"])] = r
    log_path = os.path.join(out_dir, "corun.jsonl")
    done = {}
    if os.path.exists(log_path):
        for line in open(log_path):
            r = json.loads(line)
            done[tuple(r["key"])] = r
    with open(log_path, "a") as log:
        for i, (key, r) in enumerate(sorted(recs.items())):
            if key in done:
                continue
            M, N, K, out = bucket_shape(key)
            bench = Bench(M, N, K, out, copies=2, partition=partition)
            t = corun_times(bench, r["variants"])
            rec = {"key": list(key), "shape": [M, N, K, out], "t_us": t, "flags": corun_flags(t)}
            log.write(json.dumps(rec) + "\n")
            log.flush()
            done[key] = rec
            del bench
            torch.cuda.empty_cache()
            if i % 20 == 0:
                print(f"[corun {i + 1}/{len(recs)}] {key} {t}", flush=True)
    sm_count = struct.unpack_from("<I", open(os.path.join(out_dir, "goldy_lut.bin"), "rb").read(), 20)[0]
    # preferences and flags re-derived from the logged speedups and times, so
    # the table follows the current rules
    entries = [(k, logged_pref(r), r["variants"], corun_flags(done[k]["t_us"])) for k, r in recs.items()]
    lut = write_lut(entries, G.goldy_variant_count(), sm_count)
    G.goldy_lut_from_memory(lut)
    with open(os.path.join(out_dir, "goldy_lut.bin"), "wb") as f:
        f.write(lut)
    print(f"co-run at once on {sum(1 for e in entries if e[3] & 1)} of {len(entries)} buckets", flush=True)


def rebuild_lut(profile_path: str, out_path: str, corun_path: str = None, sm_count: int = 0) -> int:
    """Re-derive a table from its profiling logs alone (no GPU): each
    bucket's preferred CD from its logged speedups under the current rule,
    its kernels as logged, its co-run flags from the logged step-3 times
    (when a co-run log is given).  The SM count comes from `sm_count` or
    from the table already at `out_path`.  Returns the number of entries."""
    recs = {}
    for line in open(profile_path):
        r = json.loads(line)
        recs[tuple(r["key"])] = r
    flags = {}
    if corun_path:
        for line in open(corun_path):
            r = json.loads(line)
            flags[tuple(r["key"])] = corun_flags(r["t_us"])
    if sm_count <= 0:
        with open(out_path, "rb") as f:
            sm_count = struct.unpack_from("<I", f.read(32), 20)[0]
    entries = [(k, logged_pref(r), r["variants"], flags.get(k, 0)) for k, r in recs.items()]
    lut = write_lut(entries, G.goldy_variant_count(), sm_count)
    G.goldy_lut_from_memory(lut)          # validate with the library's own parser
    with open(out_path, "wb") as f:
        f.write(lut)
    return len(entries)


def profile_dataset_gemm(shape, lut, log, fused: bool = True, inputs_ready: bool = False) -> dict:
    """Training record for the CD predictor (Sec. 4.3): time CD copies of one
    GEMM co-running with the table's GO-Kernel for each CD class (the kernels
    the planner would pick), CD in (1, 2, 4, 8, 16)."""
    M, N, K, out = shape
    pref, variants = G.goldy_lut_lookup(lut, G.desc(M, N, K, out))
    bench = Bench(M, N, K, out, inputs_ready=inputs_ready)
    t = {}
    for c, v in zip(CD_CLASSES, variants):
        t[c] = bench.time_us(v, c, True, target_us=1000.0, fused=fused, samples=0)
    rec = {"shape": [M, N, K, out], "variants": variants, "lut_pref_cd": pref,
           "launch": "fused" if fused else "streams", "inputs_ready": bool(inputs_ready),
           "t_us": {str(c): t[c] for c in CD_CLASSES}}
    log.write(json.dumps(rec) + "\n")
    log.flush()
    del bench
    torch.cuda.empty_cache()
    return rec


def run_dataset(path: str, total: int, lut_path: str, fused: bool, time_budget: float,
                inputs_ready: bool = False) -> int:
    done = set()
    if os.path.exists(path):
        for line in open(path):
            done.add(tuple(json.loads(line)["shape"]))
    lut = G.goldy_lut_load(lut_path)
    shapes = wl.predictor_dataset_shapes(total)
    t0 = time.time()
    with open(path, "a") as log:
        for i, sh in enumerate(shapes):
            if tuple(sh) in done:
                continue
            if time.time() - t0 > time_budget:
                print(f"time budget reached at {i} of {len(shapes)}", flush=True)
                return 0
            rec = profile_dataset_gemm(sh, lut, log, fused, inputs_ready)
            if i % 50 == 0:
                print(f"[{i + 1}/{len(shapes)}] {sh} t_us {rec['t_us']} ({time.time() - t0:.0f}s)", flush=True)
    print(f"dataset complete: {len(shapes)} GEMMs in {path}", flush=True)
    return 0


def config_keys() -> List[Tuple[int, int, int, int]]:
    keys = set()
    for name in wl.FIXED_CONFIGS:
        for s in wl.config_specs(name)[1]:
            keys.add(bucket_of(s.M, s.N, s.K, s.out_dtype))
    return sorted(keys)


def sweep_keys() -> List[Tuple[int, int, int, int]]:
    keys = set()
    for j in range(wl.SWEEP_SETS):
        for s in wl.sweep_specs(j)[1]:
            keys.add(bucket_of(s.M, s.N, s.K, s.out_dtype))
    return sorted(keys)


def bucket_of(M: int, N: int, K: int, out: int) -> Tuple[int, int, int, int]:
    key = G.goldy_bucket_key(G.desc(M, N, K, out, lda=max(8, -(-K // 8) * 8), ldb=max(8, -(-N // 8) * 8)))
    return (key >> 24) & 0xFF, (key >> 16) & 0xFF, (key >> 8) & 0xFF, key & 0xFF


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--out", default=None, help="output directory (profile.jsonl, goldy_lut.bin)")
    ap.add_argument("--dataset", default=None, metavar="JSONL",
                    help="instead of a table: time the CD predictor's training GEMMs into this file")
    ap.add_argument("--dataset-size", type=int, default=1072)
    ap.add_argument("--lut", default=G.DEFAULT_LUT, help="table whose kernels the dataset co-runs use")
    ap.add_argument("--partition", type=int, default=None, metavar="SMS",
                    help="tune inside an SM partition (green context) of at least SMS SMs (0: the whole GPU "
                         "as a partition); grid caps and the table's SM count follow the partition")
    ap.add_argument("--scaling-keys", action="store_true", help="buckets of the GPU-scaling study's sets")
    ap.add_argument("--batched-keys", action="store_true",
                    help="buckets of the batched study's B-GEMMs (M x batch rows)")
    ap.add_argument("--corun-flags", action="store_true",
                    help="step 3 over the table already profiled in --out: set each bucket's co-run flag")
    ap.add_argument("--rebuild", nargs="+", default=None, metavar=("PROFILE_JSONL", "CORUN_JSONL"),
                    help="no GPU: re-derive the table in --out (a file) from a profile log and, optionally, "
                         "a co-run log, under the current preferred-CD and co-run rules")
    ap.add_argument("--configs", action="store_true", help="buckets of the fixed workload sets")
    ap.add_argument("--sweep", action="store_true", help="buckets of the 64 randomized sets")
    ap.add_argument("--keys", nargs="*", default=[], help="extra buckets lm,ln,lk,out")
    ap.add_argument("--time-budget", type=float, default=1e9, help="stop starting buckets after this many seconds")
    ap.add_argument("--launch", choices=["fused", "streams"], default="fused",
                    help="launch mode the co-runs of step 2 use (the mode the table will be used with)")
    ap.add_argument("--top", type=int, default=1,
                    help="step 2 co-runs the best TOP kernels of each resource constraint (default 1: the paper's "
                         "single winner per constraint)")
    ap.add_argument("--inputs-ready", action="store_true",
                    help="record the timed runs with inputs_ready (a replay may overlap the previous one's tail)")
    args = ap.parse_args(argv)
    if args.dataset:
        return run_dataset(args.dataset, args.dataset_size, args.lut, args.launch == "fused", args.time_budget,
                           args.inputs_ready)
    if not args.out:
        ap.error("--out is required to build a table")
    if args.rebuild:
        n = rebuild_lut(args.rebuild[0], args.out, args.rebuild[1] if len(args.rebuild) > 1 else None)
        print(f"rebuilt {n} entries in {args.out}", flush=True)
        return 0
    if args.corun_flags:
        part = G.goldy_partition_create(args.partition, 16) if args.partition is not None else None
        add_corun_flags(args.out, args.launch == "fused", part)
        return 0
    os.makedirs(args.out, exist_ok=True)
    keys = []
    if args.configs:
        keys += config_keys()
    if args.sweep:
        keys += sweep_keys()
    if args.scaling_keys:
        keys += sorted({bucket_of(*sh) for sh in wl.scaling_study_shapes()})
    if args.batched_keys:
        keys += sorted({bucket_of(s.M * s.batch, s.N, s.K, s.out_dtype)
                        for members in (2, 4) for i in range(16) for s in wl.batched_study_specs(i, members)[1]})
    keys += [tuple(int(x) for x in k.split(",")) for k in args.keys]
    keys = sorted(set(keys))
    log_path = os.path.join(args.out, "profile.jsonl")
    done = {}
    if os.path.exists(log_path):
        for line in open(log_path):
            rec = json.loads(line)
            done[tuple(rec["key"])] = rec
    sm_count, _ = G.goldy_device_info(0)
    partition = None
    if args.partition is not None:
        partition = G.goldy_partition_create(args.partition, 16)
        sm_count = G.goldy_partition_query(partition)[0]
        print(f"profiling inside a partition of {sm_count} SMs", flush=True)
    t0 = time.time()
    with open(log_path, "a") as log:
        for i, key in enumerate(keys):
            if key in done:
                continue
            if time.time() - t0 > args.time_budget:
                print(f"time budget reached after {i} buckets", flush=True)
                break
            tb = time.time()
            rec = profile_bucket(key, sm_count, log, fused=args.launch == "fused", partition=partition,
                                 inputs_ready=args.inputs_ready, top=args.top)
            done[key] = rec
            print(f"[{i + 1}/{len(keys)}] {key} shape {rec['shape']} pref {rec['pref_cd']} "
                  f"variants {rec['variants']} ({time.time() - tb:.1f}s)", flush=True)
    entries = [(k, logged_pref(r), r["variants"]) for k, r in done.items()]
    lut = write_lut(entries, G.goldy_variant_count(), sm_count)
    G.goldy_lut_from_memory(lut)          # validate with the library's own parser
    with open(os.path.join(args.out, "goldy_lut.bin"), "wb") as f:
        f.write(lut)
    print(f"wrote {len(entries)} entries to {args.out}/goldy_lut.bin", flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())

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
         after another; the largest wins, but sequential (CD 1) unless some
         CD gains at least 5% (Sec. 5.4); CDs within 1% of the best go to the
         smaller one.

Each bucket (floor log2 of M, N, K; output dtype) is profiled at its lower
edge (M, N, K = powers of two), where DNN layer sizes usually sit.  Timing:
prepared runs (recorded plain launches, the way the benchmark replays a step)
back to back on one stream, as the paper ran GEMMs back to back on each
stream (Sec. 5.3); the median of several repetitions of a timed batch.
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


def write_lut(entries: Sequence[Tuple[Tuple[int, int, int, int], int, Sequence[int]]],
              n_variants: int, sm_count: int) -> bytes:
    """LUT bytes in the format goldy_lut_load reads (include/goldy.h)."""
    out = bytearray(b"GOLDYLUT")
    out += struct.pack("<IIIIII", 1, len(entries), n_variants, sm_count, 0, 0)
    for key, pref, variants in sorted(entries, key=lambda e: e[0]):
        out += bytes([key[0], key[1], key[2], key[3], pref, 0])
        out += struct.pack("<5H", *variants)
    return bytes(out)


def preferred_cd(speedup: Dict[int, float], gain: float = 0.05, near: float = 0.01) -> int:
    """Largest-speedup CD, sequential unless the gain reaches ``gain``; CDs
    within ``near`` of the best resolve to the smallest."""
    best_cd, best = 1, 1.0
    for cd in (2, 4, 8, 16):
        if cd in speedup and speedup[cd] > best:
            best_cd, best = cd, speedup[cd]
    if best < 1.0 + gain:
        return 1
    for cd in (2, 4, 8, 16):
        if cd in speedup and speedup[cd] >= best * (1.0 - near):
            return cd
    return best_cd


def bucket_shape(key) -> Tuple[int, int, int, int]:
    lm, ln, lk, out = key
    return 1 << lm, max(64, 1 << ln), max(64, 1 << lk), out


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
            if s > 1 and (info["cta_pair"] == 2 or s > k_blocks or tiles * s > 4 * sm_count):
                continue
            out.append((kind, s))
    return out


class Bench:
    """Buffers for up to 16 copies of one GEMM, timed through graph replays."""

    def __init__(self, M: int, N: int, K: int, out: int, copies: int = 16, seed: int = 0, partition=None,
                 graph_replay: bool = False):
        self.M, self.N, self.K, self.out = M, N, K, out
        self.partition = partition
        self.graph_replay = graph_replay
        gen = torch.Generator(device="cuda")
        gen.manual_seed(seed)
        cdt = torch.float32 if out == G.GOLDY_F32 else torch.bfloat16
        self.A = [(torch.rand((M, K), generator=gen, device="cuda") - 0.5).to(torch.bfloat16) for _ in range(copies)]
        self.B = [(torch.rand((K, N), generator=gen, device="cuda") - 0.5).to(torch.bfloat16) for _ in range(copies)]
        self.C = [torch.empty((M, N), dtype=cdt, device="cuda") for _ in range(copies)]
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
        d = G.desc(self.M, self.N, self.K, self.out)
        slots = list(range(copies)) if concurrent else [0] * copies
        sched = G.goldy_schedule_build([d] * copies, [0] * copies, [variant] * copies, slots,
                                       G.GOLDY_PLAN_FUSED if fused else 0)
        _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
        ws = self._workspace(ws_bytes)
        torch.cuda.synchronize()
        if not self.graph_replay:
            return self._time_exec(sched, copies, ws, ws_bytes, ms, target_us, samples)
        g = G.goldy_graph_create(sched, [a.data_ptr() for a in self.A[:copies]],
                                 [b.data_ptr() for b in self.B[:copies]],
                                 [c.data_ptr() for c in self.C[:copies]], ws.data_ptr(), ws_bytes,
                                 [s.cuda_stream for s in self.streams[:max(1, ms)]])
        main = self.streams[0]
        for _ in range(3 if samples else 1):
            G.goldy_graph_launch(g, main.cuda_stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(main)
        G.goldy_graph_launch(g, main.cuda_stream)
        e1.record(main)
        torch.cuda.synchronize()
        est = max(e0.elapsed_time(e1) * 1e3, 1.0)
        if samples == 0:                 # quick mode: one replay is long enough to time on its own
            if est >= target_us:
                return est
            samples = 3
        reps = int(min(200, max(3, target_us / est)))
        times = []
        for _ in range(samples):
            e0.record(main)
            for _ in range(reps):
                G.goldy_graph_launch(g, main.cuda_stream)
            e1.record(main)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1) * 1e3 / reps)
        if G.goldy_device_error(clear=True) != 0:
            raise RuntimeError("kernel reported a bounded-wait timeout while profiling")
        times.sort()
        return times[len(times) // 2]


def profile_bucket(key, sm_count: int, log, fused: bool = True, partition=None) -> dict:
    M, N, K, out = bucket_shape(key)
    bench = Bench(M, N, K, out, partition=partition)
    cands = candidates(M, N, K, sm_count)
    rows = []
    winners = {}
    for rc in RC_DIVS:                                  # step 1
        best = None
        for kind, split in cands:
            v = G.variant_id(kind, split, rc)
            t = bench.time_us(v, 1, True, fused=fused)
            rows.append({"step": 1, "rc": rc, "variant": v, "us": t})
            if best is None or t < best[0]:
                best = (t, v)
        winners[rc] = best
    go = {1: winners[1][1]}
    t_cd = {1: winners[1][0]}
    for cd in (2, 4, 8, 16):                            # step 2
        best = None
        for rc in RC_DIVS:
            v = winners[rc][1]
            t = bench.time_us(v, cd, True, fused=fused)
            rows.append({"step": 2, "cd": cd, "rc": rc, "variant": v, "us": t})
            if best is None or t < best[0]:
                best = (t, v)
        go[cd] = best[1]
        t_cd[cd] = best[0]
    speedup = {cd: cd * t_cd[1] / t_cd[cd] for cd in CD_CLASSES}
    pref = preferred_cd(speedup)
    rec = {"key": list(key), "shape": [M, N, K, out], "pref_cd": pref, "launch": "fused" if fused else "streams",
           "variants": [go[c] for c in CD_CLASSES], "t_us": {str(c): t_cd[c] for c in CD_CLASSES},
           "speedup": {str(c): speedup[c] for c in CD_CLASSES}, "rows": rows}
    log.write(json.dumps(rec) + "\n")
    log.flush()
    del bench
    torch.cuda.empty_cache()
    return rec


def _time_exec(self, sched, copies, ws, ws_bytes, ms, target_us, samples):
    """time_us as prepared runs (recorded plain launches) replayed back to back
    on the bench's streams — or the partition's — and timed by events on the
    first of them (goldy_exec_time)."""
    x = G.goldy_exec_create(sched, [a.data_ptr() for a in self.A[:copies]], [b.data_ptr() for b in self.B[:copies]],
                            [c.data_ptr() for c in self.C[:copies]], ws.data_ptr(), ws_bytes,
                            self.part_streams[:max(1, ms)])
    est = max(G.goldy_exec_time([x], 3 if samples else 1, 1) * 1e3, 1.0)
    if samples == 0:
        if est >= target_us:
            return est
        samples = 3
    reps = int(min(200, max(3, target_us / est)))
    times = sorted(G.goldy_exec_time([x], 0, reps) * 1e3 for _ in range(samples))
    del x
    if G.goldy_device_error(clear=True) != 0:
        raise RuntimeError("kernel reported a bounded-wait timeout while profiling")
    return times[len(times) // 2]


Bench._time_exec = _time_exec


def profile_dataset_gemm(shape, lut, log, fused: bool = True) -> dict:
    """Training record for the CD predictor (Sec. 4.3): time CD copies of one
    GEMM co-running with the table's GO-Kernel for each CD class (the kernels
    the planner would pick), CD in (1, 2, 4, 8, 16)."""
    M, N, K, out = shape
    pref, variants = G.goldy_lut_lookup(lut, G.desc(M, N, K, out))
    bench = Bench(M, N, K, out)
    t = {}
    for c, v in zip(CD_CLASSES, variants):
        t[c] = bench.time_us(v, c, True, target_us=1000.0, fused=fused, samples=0)
    rec = {"shape": [M, N, K, out], "variants": variants, "lut_pref_cd": pref,
           "launch": "fused" if fused else "streams", "t_us": {str(c): t[c] for c in CD_CLASSES}}
    log.write(json.dumps(rec) + "\n")
    log.flush()
    del bench
    torch.cuda.empty_cache()
    return rec


def run_dataset(path: str, total: int, lut_path: str, fused: bool, time_budget: float) -> int:
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
            rec = profile_dataset_gemm(sh, lut, log, fused)
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
    ap.add_argument("--configs", action="store_true", help="buckets of the fixed workload sets")
    ap.add_argument("--sweep", action="store_true", help="buckets of the 64 randomized sets")
    ap.add_argument("--keys", nargs="*", default=[], help="extra buckets lm,ln,lk,out")
    ap.add_argument("--time-budget", type=float, default=1e9, help="stop starting buckets after this many seconds")
    ap.add_argument("--launch", choices=["fused", "streams"], default="fused",
                    help="launch mode the co-runs of step 2 use (the mode the table will be used with)")
    args = ap.parse_args(argv)
    if args.dataset:
        return run_dataset(args.dataset, args.dataset_size, args.lut, args.launch == "fused", args.time_budget)
    if not args.out:
        ap.error("--out is required to build a table")
    os.makedirs(args.out, exist_ok=True)
    keys = []
    if args.configs:
        keys += config_keys()
    if args.sweep:
        keys += sweep_keys()
    if args.scaling_keys:
        keys += sorted({bucket_of(*sh) for sh in wl.scaling_study_shapes()})
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
            rec = profile_bucket(key, sm_count, log, fused=args.launch == "fused", partition=partition)
            done[key] = rec
            print(f"[{i + 1}/{len(keys)}] {key} shape {rec['shape']} pref {rec['pref_cd']} "
                  f"variants {rec['variants']} ({time.time() - tb:.1f}s)", flush=True)
    entries = [(k, r["pref_cd"], r["variants"]) for k, r in done.items()]
    lut = write_lut(entries, G.goldy_variant_count(), sm_count)
    G.goldy_lut_from_memory(lut)          # validate with the library's own parser
    with open(os.path.join(args.out, "goldy_lut.bin"), "wb") as f:
        f.write(lut)
    print(f"wrote {len(entries)} entries to {args.out}/goldy_lut.bin", flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())

#!/usr/bin/env python
"""Concurrent-GEMM set benchmark on GB300.

One step = one pass of the whole hot path over one synthetic GEMM set: the
dynamic logic's plan (computed once; it is a pure function of the shapes)
replayed as a prepared run of GO-Kernel launches on CD streams (recorded
once, replayed with plain launches; ``--replay graph`` replays a captured
CUDA graph instead).  Default workload: the heterogeneous pair of two
co-running models, 3 GEMMs of M=512, N=1024, K=1024 plus one of M=2048,
N=8192, K=2048, bf16 in, fp32 accumulate and out — the largest fixed set and
the compute-bound one.  The other fixed sets are measured on the same line
as extra keys.

Prints ONE JSON line (rank 0): TFLOP/s of the whole job (all ranks), the
makespan, speedups over sequential and naive all-streams execution of the
same library, cuBLAS as a reference point, a roofline entry for the dominant
kernel, the CPU oracle as a baseline, clocks sampled during the timed region,
and an end-to-end number through host buffers.

Multi-GPU: a set of independent GEMMs needs no exchange, so N ranks run N
independent replicas (weak scaling, no collective on the data path); the
only collectives are the barrier and the max-reduction of the timed region.

``--impl reference`` times the CPU oracle (test infrastructure) on the same
workload instead, on the host's cores, rank 0 only.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "concurrent-GEMM set TFLOP/s and makespan speedup vs sequential and naive streams"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
CSRC = os.path.join(ROOT, "paper_2409_02227_gb300", "csrc")


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description="concurrent-GEMM set benchmark")
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=["goldy", "reference"], default="goldy")
    ap.add_argument("--config", default="hetero_pair",
                    help="workload: pair_256, ffn_slices, lstm_gates, hetero_pair or sweep_00 .. sweep_63")
    ap.add_argument("--extra-configs", default="pair_256,ffn_slices,lstm_gates",
                    help="comma-separated fixed sets also measured on the line ('' for none)")
    ap.add_argument("--lut", default=None, help="lookup table (default: the packaged one)")
    ap.add_argument("--launch", choices=["fused", "streams"], default="fused",
                    help="fused: a wave's same-kind GEMMs share one launch; streams: one launch per GEMM")
    ap.add_argument("--replay", choices=["exec", "graph"], default="exec",
                    help="how the prepared step is replayed: recorded plain launches or a CUDA graph")
    ap.add_argument("--serial-launch", action="store_true",
                    help="plain serialised launches (no overlap of a launch's set-up with the previous kernel)")
    ap.add_argument("--no-inputs-ready", action="store_true",
                    help="do not let a launch's loads and MMAs start during the previous kernel's tail "
                         "(goldy_run_opts.inputs_ready = 0)")
    ap.add_argument("--soak", type=float, default=1.0,
                    help="seconds of the same steps run right before the timed region (sustained clocks)")
    ap.add_argument("--no-compare", action="store_true", help="skip sequential/naive/cuBLAS comparisons")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--batched-study", default=None, metavar="FILE",
                    help="heterogeneous strided-batched GEMM study (JSON to FILE)")
    ap.add_argument("--corun-study", default=None, metavar="FILE",
                    help="GEMM + element-wise add co-scheduling study (JSON to FILE)")
    ap.add_argument("--scaling-study", default=None, metavar="FILE",
                    help="GPU-scaling study inside SM partitions of 1/4, 1/2 and all of the GPU (JSON to FILE)")
    ap.add_argument("--phase-trace", action="store_true",
                    help="instead of the JSON line: per-launch phase times (device trace) of one step of the "
                         "planned set, replayed among back-to-back steps (markdown on stdout)")
    ap.add_argument("--report", default=None, metavar="FILE",
                    help="instead of the JSON line: time every fixed set and the 64 randomized sets "
                         "under every policy and write a JSON report to FILE (markdown table on stdout)")
    return ap.parse_args(argv)


# ----------------------------------------------------------------------------- distributed
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return world, rank, local


def dist_init(world: int, backend: str):
    if world <= 1:
        return None
    import torch.distributed as dist
    if not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def reduce_max(value: float, dist, device=None) -> float:
    """Max of `value` over ranks (the slowest rank sets the job's time)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist, device=None):
    if dist is not None:
        if device is not None:
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock / throttle-reason samples (100 ms) around the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index                 # nvidia-smi --id: PCI bus id or index
        self.samples = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=5)

    def summary(self, t0: float, t1: float) -> dict:
        win = [s for t, s in self.samples if t0 - 0.15 <= t <= t1 + 0.15]
        if not win:
            win = [s for _, s in self.samples]
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(s[1]) for s in win if s[1].replace(".", "").isdigit()]
        mx = [float(s[2]) for s in win if s[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for s in win:
            for name, v in zip(names, s[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(win)}


# ----------------------------------------------------------------------------- helpers
def peaks():
    try:
        with open(PEAKS_FILE) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, 1900.0, 1700.0, "fallback"


KERNEL_SOURCES = ("go_kernel.cuh", "go_kernel_pair.cuh", "sm103_ptx.cuh", "kernels.cu", "goldy_internal.h")


def csrc_hash() -> str:
    """Hash of the device-code sources: a recorded DRAM traffic figure is
    only used while the kernels it was measured on are unchanged."""
    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(name.encode())
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(variant_name: str):
    """DRAM bytes per launch from a committed ncu capture, if it was taken on
    the current kernel source and the same variant; else None."""
    try:
        with open(TRAFFIC_FILE) as f:
            t = json.load(f)
    except (OSError, ValueError):
        return None
    h = csrc_hash()
    for e in t.get("entries", []):
        if e.get("csrc_hash") == h and e.get("variant") == variant_name:
            return e.get("dram_bytes_per_launch")
    return None


def workload_label(specs) -> str:
    from collections import Counter
    c = Counter((s.M, s.N, s.K, "bf16" if s.out_dtype == 0 else "fp32") for s in specs)
    return " + ".join(f"{n}x(M={m},N={nn},K={k},{o} out)" for (m, nn, k, o), n in c.items())


def load_set(name: str):
    """A fixed workload set by name, or randomized set j as sweep_jj."""
    from paper_2409_02227_gb300 import workloads as wl
    if name.startswith("sweep_"):
        return wl.make_sweep_set(int(name.split("_")[1]))
    return wl.make_config(name)


# ----------------------------------------------------------------------------- CPU oracle
def oracle_sample(st, budget_s: float):
    """Run the fp64 oracle over GEMMs of the set (whole GEMMs, in order,
    cycling) until about `budget_s` of work is done; returns
    (flops, seconds, threads, description)."""
    from oracle import gemm as og
    flops = 0
    done = []
    t0 = time.perf_counter()
    i = 0
    while True:
        og.gemm(st.a_bits(i % len(st.specs)), st.b_bits(i % len(st.specs)))
        flops += st.specs[i % len(st.specs)].flops
        done.append(i % len(st.specs))
        i += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    desc = f"{len(done)} whole GEMMs of the set (indices {done[:8]}{'...' if len(done) > 8 else ''}), fp64 oracle"
    return flops, dt, og.num_threads(), desc


def run_reference(args, world, rank):
    """Reference arm: the CPU oracle timed on the host's cores."""
    if rank != 0:
        return 0
    from oracle import gemm as og
    st = load_set(args.config)
    # each step computes a fixed number of output entries of every GEMM of the
    # set (exact fp64 dot products), sized so the whole run takes about a minute
    import numpy as np
    K, W = max(1, args.steps), max(0, args.warmup)

    def pick(i, n, step):
        sp = st.specs[i]
        r = np.random.default_rng([step + 1000, i])
        return r.integers(0, sp.M, n), r.integers(0, sp.N, n)

    t0 = time.perf_counter()
    for i in range(len(st.specs)):
        ii, jj = pick(i, 64, -1)
        og.gemm_entries(st.a_bits(i), st.b_bits(i), ii, jj)
    per_entry = max((time.perf_counter() - t0) / 64, 1e-7)
    entries = int(max(1, min(4096, 60.0 / (K + W) / per_entry)))
    flops_step = sum(2 * entries * s.K for s in st.specs)
    for step in range(-W, K):
        if step == 0:
            t0 = time.perf_counter()
        for i in range(len(st.specs)):
            ii, jj = pick(i, entries, step)
            og.gemm_entries(st.a_bits(i), st.b_bits(i), ii, jj)
    dt = time.perf_counter() - t0
    value = flops_step * K / dt / 1e12
    sample = (f"{entries} seeded random output entries of each of the {len(st.specs)} GEMMs per step "
              f"(exact fp64 dot products over the full K)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": dt / K * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{args.config}: {workload_label(st.specs)}", "sample": sample},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": og.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- GPU arm
def c_shape(s):
    """Shape of a GEMM's output (entries first for a strided batch)."""
    return (s.M, s.N) if s.batch == 1 else (s.batch, s.M, s.N)


class SetRunner:
    """R rotating device copies of one GEMM set, each with its run prepared
    once: a recorded prepared run (``replay="exec"``, plain launches) or a
    captured CUDA graph (``replay="graph"``).  Construction replays every
    prepared run once (untimed), so none is first launched inside a timed
    region."""

    def __init__(self, st, sched, copies, with_events=False, replay="exec", serial_launch=False, inputs_ready=True):
        import torch
        from paper_2409_02227_gb300 import goldy as G
        self.G = G
        self.torch = torch
        self.sched = sched
        self.replay = replay
        n, _, ms, ws_bytes = G.goldy_schedule_query(sched)
        self.n = n
        self.ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
        self.ws_bytes = ws_bytes
        self.streams = [torch.cuda.Stream() for _ in range(max(1, ms))]
        base_a = [a.cuda() for a in st.a]
        base_b = [b.cuda() for b in st.b]
        cdt = [torch.bfloat16 if s.out_dtype == 0 else torch.float32 for s in st.specs]
        self.copies = []
        for r in range(copies):
            A = base_a if r == 0 else [a.clone() for a in base_a]
            B = base_b if r == 0 else [b.clone() for b in base_b]
            C = [torch.empty(c_shape(s), dtype=d, device="cuda") for s, d in zip(st.specs, cdt)]
            self.copies.append((A, B, C))
        self.events = []
        self.runs = []
        torch.cuda.synchronize()
        sp = [s.cuda_stream for s in self.streams]
        for A, B, C in self.copies:
            ptrs = ([a.data_ptr() for a in A], [b.data_ptr() for b in B], [c.data_ptr() for c in C])
            evs = {}
            if with_events:
                eb = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
                ee = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
                for e in eb + ee:            # torch creates the CUDA event on first record
                    e.record()
                torch.cuda.synchronize()
                evs = {"ev_begin": [e.cuda_event for e in eb], "ev_end": [e.cuda_event for e in ee]}
                self.events.append((eb, ee))
            # inputs_ready: no kernel of the run writes an A or B (each step
            # reads its own copy, written once before any step), so the load
            # and MMA roles may start during the previous kernel's tail
            if replay == "exec":
                r = G.goldy_exec_create(sched, *ptrs, self.ws.data_ptr(), ws_bytes, sp, serial_launch=serial_launch,
                                        inputs_ready=inputs_ready, **evs)
            else:
                r = G.goldy_graph_create_ex(sched, *ptrs, self.ws.data_ptr(), ws_bytes, sp,
                                            evs.get("ev_begin"), evs.get("ev_end"), serial_launch=serial_launch,
                                            inputs_ready=inputs_ready)
            self.runs.append(r)
        self.main = self.streams[0]
        for k in range(len(self.runs)):
            self.launch(k)
        torch.cuda.synchronize()

    def __del__(self):
        # destroy the prepared runs before the buffers they read and write
        self.runs.clear()

    def launch(self, k):
        r = self.runs[k % len(self.runs)]
        if self.replay == "exec":
            self.G.goldy_exec_launch(r)
        else:
            self.G.goldy_graph_launch(r, self.main.cuda_stream)

    def spin(self, us):
        """Keep the launching stream busy for about `us` microseconds (a
        clock-cycle spin kernel) so that the host has queued what follows
        before the GPU reaches it: a timed region then measures the device,
        not the host's launch rate."""
        torch = self.torch
        with torch.cuda.stream(self.main):
            torch.cuda._sleep(int(us * 2000))

    def timed(self, steps, spin_us=200.0):
        """Elapsed ms of `steps` back-to-back replays (copy k % R for step k),
        bracketed by one event pair on the launching stream and nothing in
        between."""
        torch = self.torch
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        self.spin(spin_us)
        e0.record(self.main)
        for k in range(steps):
            self.launch(k)
        e1.record(self.main)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    def step_distribution(self, reps, mode, flush=None, spin_us=25.0):
        """Per-step device time over `reps` single steps, each bracketed by its
        own event pair: ``cold`` flushes the L2 (writes `flush`, a buffer of
        twice its size) and rotates the copies before each step; ``warm``
        replays copy 0 untimed right before each timed replay of copy 0, so
        its operands sit in the L2.  A short spin before each timed step lets
        the host queue the step first.  Median, p10 and p90 in us."""
        torch = self.torch
        pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for i, (a, b) in enumerate(pairs):
            if mode == "cold":
                with torch.cuda.stream(self.main):
                    flush.zero_()
                k = i
            else:
                self.launch(0)
                k = 0
            self.spin(spin_us)
            a.record(self.main)
            self.launch(k)
            b.record(self.main)
        torch.cuda.synchronize()
        return percentiles([a.elapsed_time(b) * 1e3 for a, b in pairs])

    def launch_durations_ms(self):
        out = []
        for eb, ee in self.events:
            for b, e in zip(eb, ee):
                out.append(b.elapsed_time(e))
        return out


def percentiles(xs):
    xs = sorted(xs)
    q = lambda f: xs[min(len(xs) - 1, max(0, int(round(f * (len(xs) - 1)))))]
    return {"median_us": q(0.5), "p10_us": q(0.1), "p90_us": q(0.9), "reps": len(xs)}


def soak(runner, seconds):
    """About `seconds` of the runner's steps back to back (untimed), so that
    the clocks a following timed region runs at are those of this load."""
    if seconds <= 0:
        return
    est_ms = max(1e-3, runner.timed(20) / 20)
    runner.timed(int(min(200000, max(20, seconds * 1e3 / est_ms))))


def time_schedule(st, sched, copies, steps, soak_s=0.0):
    """Makespan (us) of one schedule, replayed both ways (recorded plain
    launches and a CUDA graph); each configuration is credited with its
    faster replay, so that no baseline is slowed by a launch mode that does
    not suit it.  With `soak_s`, each timed region follows that long of the
    same steps (sustained clocks, as the bench line's own region).  Returns
    (best, {"exec": us, "graph": us})."""
    import torch
    out = {}
    for mode in ("exec", "graph"):
        r = SetRunner(st, sched, copies, replay=mode)
        for k in range(10):
            r.launch(k)
        torch.cuda.synchronize()
        soak(r, soak_s)
        out[mode] = r.timed(steps) / steps * 1e3
        del r
    return min(out.values()), out


def cublas_reference_ms(st, copies, steps):
    """torch.matmul (cuBLAS) for the same set, as a reference point only:
    ``sequential`` runs the set's GEMMs back to back on one stream;
    ``streams`` forks one stream per GEMM from the launching stream and joins
    them back (the naive all-streams launch).  Each is one CUDA graph that
    runs the set once per rotating copy (so the inputs come from HBM),
    replayed after ~0.3 s of the same replays; ms per set."""
    import torch
    base_a = [a.cuda() for a in st.a]
    base_b = [b.cuda() for b in st.b]
    s = torch.cuda.Stream()
    side = [torch.cuda.Stream() for _ in st.a]
    keep = []                   # the captured graphs read every copy: keep them all alive
    for r in range(copies):
        A = base_a if r == 0 else [a.clone() for a in base_a]
        B = base_b if r == 0 else [b.clone() for b in base_b]
        keep.append((A, B))
    for st_ in [s] + side:
        with torch.cuda.stream(st_):
            for a, b in zip(*keep[0]):
                torch.matmul(a, b)      # warm cuBLAS handles on every stream outside the capture
    torch.cuda.synchronize()
    out = {}
    for mode in ("sequential", "streams"):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            outs = []
            for A, B in keep:
                if mode == "sequential":
                    outs.append([torch.matmul(a, b) for a, b in zip(A, B)])
                    continue
                for x in side:
                    x.wait_stream(s)
                row = []
                for x, a, b in zip(side, A, B):
                    with torch.cuda.stream(x):
                        row.append(torch.matmul(a, b))
                for x in side:
                    s.wait_stream(x)
                outs.append(row)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        # ~0.3 s of the same replays first (sustained clocks, like every
        # other configuration on the line)
        q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        q0.record()
        for _ in range(3):
            g.replay()
        q1.record()
        torch.cuda.synchronize()
        per_ms = max(1e-3, q0.elapsed_time(q1) / 3)
        for _ in range(int(min(20000, 300.0 / per_ms))):
            g.replay()
        reps = max(3, steps // copies)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
        out[mode] = e0.elapsed_time(e1) / (reps * copies)
        del g, outs
    del keep
    return out


def e2e_measure(st, sched, steps):
    """Same metric through host buffers and the public API: every step copies
    its A and B from pinned host memory, runs goldy_run, and reads its C back
    to pinned host memory.  Steps are pipelined the way a serving loop would
    run them: two device buffer sets, input copies on one copy stream, the
    GEMMs on the run's streams, result copies on another copy stream, ordered
    by events, so step k's input copy overlaps step k-1's GEMMs and step
    k-2's result copy.  Also times the copies alone (same bytes, same
    pipeline, no GEMMs): the ceiling the end-to-end number can reach on this
    host link."""
    import torch
    from paper_2409_02227_gb300 import goldy as G
    _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
    streams = [torch.cuda.Stream() for _ in range(max(1, ms))]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    hA = [a.pin_memory() for a in st.a]
    hB = [b.pin_memory() for b in st.b]
    cdt = [torch.bfloat16 if s.out_dtype == 0 else torch.float32 for s in st.specs]
    hC = [[torch.empty(c_shape(s), dtype=d).pin_memory() for s, d in zip(st.specs, cdt)] for _ in range(2)]
    dA = [[torch.empty_like(a, device="cuda") for a in st.a] for _ in range(2)]
    dB = [[torch.empty_like(b, device="cuda") for b in st.b] for _ in range(2)]
    dC = [[torch.empty(c_shape(s), dtype=d, device="cuda") for s, d in zip(st.specs, cdt)] for _ in range(2)]
    main = streams[0]
    sp = [s.cuda_stream for s in streams]
    ev = lambda: torch.cuda.Event()
    in_done = [ev(), ev()]
    gemm_done = [ev(), ev()]
    out_done = [ev(), ev()]
    for e in in_done + gemm_done + out_done:
        e.record(main)                       # created and complete: the first waits pass

    def step(k, gemm=True):
        b = k % 2
        s_in.wait_event(gemm_done[b])        # the GEMMs of step k-2 have read this buffer set
        with torch.cuda.stream(s_in):
            for d, h in zip(dA[b] + dB[b], hA + hB):
                d.copy_(h, non_blocking=True)
        in_done[b].record(s_in)
        main.wait_event(in_done[b])
        main.wait_event(out_done[b])         # step k-2's results have left this buffer set
        if gemm:
            G.goldy_run(sched, [a.data_ptr() for a in dA[b]], [x.data_ptr() for x in dB[b]],
                        [c.data_ptr() for c in dC[b]], ws.data_ptr(), ws_bytes, sp)
        gemm_done[b].record(main)
        s_out.wait_event(gemm_done[b])
        with torch.cuda.stream(s_out):
            for h, d in zip(hC[b], dC[b]):
                h.copy_(d, non_blocking=True)
        out_done[b].record(s_out)

    def run(gemm):
        for k in range(4):
            step(k, gemm)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(main)
        s_in.wait_stream(main)
        for k in range(steps):
            step(k, gemm)
        main.wait_stream(s_out)
        e1.record(main)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps

    ms_step = run(True)
    ms_copies = run(False)
    h2d = sum(a.numel() * a.element_size() for a in hA + hB)
    d2h = sum(c.numel() * c.element_size() for c in hC[0])
    return ms_step, ms_copies, h2d, d2h


def plan_set(G, st, lut, launch_flag):
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype, batch=s.batch) for s in st.specs]
    sched = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | launch_flag)
    plan = [G.goldy_schedule_entry(sched, i) for i in range(len(descs))]
    kinds = {(G.goldy_variant_info_get(v)["kind"], st.specs[i].out_dtype) for i, (_, v, _, _) in enumerate(plan)}
    n_groups = G.goldy_schedule_query(sched)[1]
    single = bool(launch_flag) and n_groups == 1 and len(kinds) == 1 and plan[0][3] >= len(descs)
    return descs, sched, plan, single


def rotating_copies(st, l2):
    in_bytes = sum(s.batch * (2 * s.M * s.K + 2 * s.K * s.N) for s in st.specs)
    return max(2, math.ceil(2 * l2 / in_bytes)), in_bytes


def compare_policies(G, st, descs, lut, copies, csteps, launch_flag, soak_s=0.3):
    """Every policy timed like the bench line's own region: prepared runs (or
    graphs) over the rotating copies, back to back after ~soak_s seconds of
    the same steps; cuBLAS, timed the same way, as a reference point."""
    comp, modes = {}, {}
    for name, flags in (("sequential", G.GOLDY_PLAN_SEQUENTIAL), ("naive_streams", G.GOLDY_PLAN_DEFAULT),
                        ("go_all_concurrent", G.GOLDY_PLAN_GO),
                        ("goldyloc_streams", G.GOLDY_PLAN_AUTO),
                        ("goldyloc_fused", G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)):
        s2 = G.goldy_plan(descs, lut, flags)
        comp[name], modes[name] = time_schedule(st, s2, copies, csteps, soak_s)
    a_us = comp["goldyloc_fused" if launch_flag else "goldyloc_streams"]
    cb = cublas_reference_ms(st, copies, csteps)
    out = {"comparisons_us": {**comp, "cublas_sequential_reference": cb["sequential"] * 1e3,
                              "cublas_streams_reference": cb["streams"] * 1e3, "by_replay": modes,
                              "note": "each configuration at its faster replay (recorded launches or graph), "
                                      "timed after ~0.3 s of its own steps (sustained clocks, like the line's own "
                                      "region); cuBLAS (torch.matmul, timed the same way) is a reference point only"},
           "speedup_vs_sequential": comp["sequential"] / a_us,
           "speedup_vs_naive_streams": comp["naive_streams"] / a_us}
    return out


def roof_of(st, us, hbm, tf_burst, tf_sust):
    roof_us = max(st.flops / (tf_burst * 1e12), st.bytes / (hbm * 1e9)) * 1e6
    bound = "tensor" if st.flops / st.bytes > tf_burst * 1e12 / (hbm * 1e9) else "hbm"
    out = {"bound": bound, "set_roof_us": roof_us, "frac": roof_us / us}
    if bound == "tensor":
        out["frac_sustained"] = st.flops / (tf_sust * 1e12) * 1e6 / us
    return out


def measure_extra(G, name, lut, l2, launch_flag, flush, steps, peaks_):
    """One more fixed set on the bench line: its planned step replayed back to
    back (long run), per-step distributions L2-cold and warm, comparisons."""
    import torch
    from paper_2409_02227_gb300 import workloads as wl
    hbm, tf_burst, tf_sust = peaks_
    st = wl.make_config(name)
    descs, sched, plan, single = plan_set(G, st, lut, launch_flag)
    copies, _ = rotating_copies(st, l2)
    r = SetRunner(st, sched, copies)
    cold = r.step_distribution(100, "cold", flush)
    warm = r.step_distribution(100, "warm")
    soak(r, 0.3)
    us = r.timed(steps) / steps * 1e3
    del r
    torch.cuda.synchronize()
    out = {"workload": workload_label(st.specs), "makespan_us": us, "tflops": st.flops / (us * 1e-6) / 1e12,
           "steps": steps, "step_cold_us": cold, "step_warm_us": warm,
           "plan": [G.goldy_variant_info_get(v)["name"] for _, v, _, _ in plan],
           "launches_per_step": 1 if single else len(plan),
           "roofline": roof_of(st, us, hbm, tf_burst, tf_sust)}
    out.update(compare_policies(G, st, descs, lut, copies, max(200, min(steps, 2000)), launch_flag))
    return out


def run_gpu(args, world, rank, local):
    import torch
    dist = dist_init(world, "nccl")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    from paper_2409_02227_gb300 import goldy as G
    from paper_2409_02227_gb300 import workloads as wl

    st = load_set(args.config)
    lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    launch_flag = G.GOLDY_PLAN_FUSED if args.launch == "fused" else 0
    descs, sched, plan, single_launch = plan_set(G, st, lut, launch_flag)
    props = torch.cuda.get_device_properties(device)
    l2 = int(getattr(props, "L2_cache_size", 126 * 1024 * 1024))
    copies, in_bytes = rotating_copies(st, l2)
    flush = torch.empty(2 * l2, dtype=torch.uint8, device="cuda")
    hbm, tf_burst, tf_sust, peak_src = peaks()

    # every prepared run is replayed once while the runner is built
    ready = not args.no_inputs_ready
    runner = SetRunner(st, sched, copies, replay=args.replay, serial_launch=args.serial_launch, inputs_ready=ready)
    try:
        gpu_id = "%08X:%02X:%02X.0" % (props.pci_domain_id, props.pci_bus_id, props.pci_device_id)
    except AttributeError:
        gpu_id = str(local)
    sampler = ClockSampler(gpu_id)
    sampler.start()
    t_load0 = time.time()
    # per-step distributions (separate passes, never inside the headline
    # region), then a second of the same back-to-back steps so that the
    # clocks sampled around the timed region are those of this load
    cold = runner.step_distribution(200, "cold", flush)
    warm = runner.step_distribution(200, "warm")
    est_us = max(1.0, cold["median_us"])
    soak_steps = int(min(200000, max(20, args.soak * 1e6 / est_us)))
    runner.timed(soak_steps)
    for k in range(args.warmup):
        runner.launch(k)
    torch.cuda.synchronize()
    barrier(dist, device)
    torch.cuda.synchronize()
    t_wall0 = time.time()
    elapsed_ms = runner.timed(args.steps)
    t_wall1 = time.time()
    barrier(dist, device)
    sampler.stop()
    elapsed_ms = reduce_max(elapsed_ms, dist, device)
    if G.goldy_device_error(clear=True) != 0:
        raise RuntimeError("a GO-Kernel reported a bounded-wait timeout during the timed region")
    ms_step = elapsed_ms / args.steps
    value = world * st.flops / (ms_step * 1e-3) / 1e12

    # dominant kernel: the variant carrying the most FLOPs in the plan
    by_variant = {}
    for i, (g, v, slot, cd) in enumerate(plan):
        by_variant.setdefault(v, []).append(i)
    dom_v = max(by_variant, key=lambda v: sum(st.specs[i].flops for i in by_variant[v]))
    dom_idx = by_variant[dom_v]
    if single_launch:
        # one launch per step, covering all GEMMs, on the launching stream:
        # its average duration is the timed region's elapsed time over the
        # steps (back-to-back launches, so an upper bound)
        durs = [ms_step]
        dom_idx = list(range(len(descs)))
        timing_note = ("CUDA events on the launching stream around the timed region / steps "
                       "(one launch per step, launches back to back)")
    else:
        inst = SetRunner(st, sched, copies, with_events=True, replay=args.replay, serial_launch=args.serial_launch,
                         inputs_ready=ready)
        for k in range(2 * copies):
            inst.launch(k)
        torch.cuda.synchronize()
        durs = [eb[i].elapsed_time(ee[i]) for eb, ee in inst.events for i in dom_idx]
        del inst
        timing_note = "events recorded around each launch on its own stream inside an instrumented copy of the run"
    dur_ms = statistics.mean(durs)
    bytes_per_launch = sum(st.specs[i].bytes for i in dom_idx) / (1 if single_launch else len(dom_idx))
    flops_per_launch = sum(st.specs[i].flops for i in dom_idx) / (1 if single_launch else len(dom_idx))
    ai = flops_per_launch / bytes_per_launch
    ridge = tf_burst * 1e12 / (hbm * 1e9)
    vname = G.goldy_variant_info_get(dom_v)["name"] + (f" fused x{len(descs)}" if single_launch else "")
    if ai < ridge:
        achieved = bytes_per_launch / (dur_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm}
    else:
        achieved = flops_per_launch / (dur_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": tf_burst, "unit": "TFLOP/s",
                "frac": achieved / tf_burst, "peak_sustained": tf_sust, "frac_sustained": achieved / tf_sust}
    roof["traffic"] = recorded_traffic(vname)
    roof.update({"kernel": vname, "launch_us": dur_ms * 1e3,
                 "launches_sampled": args.steps if single_launch else len(durs),
                 "timing": timing_note,
                 "per_launch": {"algorithmic_bytes": bytes_per_launch, "flops": flops_per_launch},
                 "peak_source": f"{peak_src} ({'HBM copy' if roof['bound'] == 'hbm' else 'cuBLAS bf16 burst; sustained beside it'})"})

    set_roof = roof_of(st, ms_step * 1e3, hbm, tf_burst, tf_sust)
    launches_per_step = 1 if single_launch else sum(1 for s in st.specs if s.M and s.N and s.K)
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{args.config}: {workload_label(st.specs)}",
                   "l2": f"inputs larger than L2: {copies} rotating device copies of the set "
                         f"({copies * in_bytes / 2**20:.0f} MiB of A/B vs {l2 / 2**20:.0f} MiB L2); "
                         f"no flush inside the timed region",
                   "launch": f"{'prepared-run' if args.replay == 'exec' else 'CUDA graph'} replay of the planned "
                             f"schedule ({args.launch} launch mode, "
                             f"{'serialised launches' if args.serial_launch else 'each launch set-up overlapping the previous kernel (programmatic dependent launch)'}"
                             f"{'' if args.serial_launch or not ready else '; loads and MMAs of a launch may start during the previous kernel, its stores only after it (inputs_ready: no kernel writes an A or B)'}); "
                             f"the timed region is one event pair around the steps, queued behind a 200 us spin "
                             f"so the host has issued them before the GPU reaches them",
                   "plan": [{"gemm": i, "group": g, "variant": G.goldy_variant_info_get(v)["name"], "slot": sl,
                             "cd": cd} for i, (g, v, sl, cd) in enumerate(plan)],
                   "parallelism": f"replicas x{world}"},
        "makespan_us": ms_step * 1e3,
        "set_roof_us": set_roof["set_roof_us"],
        "set_roofline_frac": set_roof["frac"],
        "step_cold_us": cold,
        "step_warm_us": warm,
        "soak_steps_before_timing": soak_steps,
        "gpu_launches": launches_per_step * args.steps,
        "roofline": roof,
    }
    clocks = sampler.summary(t_load0, t_wall1)
    clocks["window"] = "per-step passes, the soak and the timed region"
    line["clocks"] = clocks

    if not args.no_compare:
        line.update(compare_policies(G, st, descs, lut, copies, max(200, min(args.steps, 5000)), launch_flag))

    e2e_steps = max(5, min(args.steps, 200))
    e_ms, c_ms, h2d, d2h = e2e_measure(st, sched, e2e_steps)
    e_ms = reduce_max(e_ms, dist, device)
    line["e2e"] = {"value": world * st.flops / (e_ms * 1e-3) / 1e12, "unit": "TFLOP/s",
                   "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms,
                   "steps": e2e_steps,
                   "copies_alone_ms_per_step": c_ms,
                   "copies_alone_gbs": (h2d + d2h) / (c_ms * 1e-3) / 1e9,
                   "pipeline": "two buffer sets; step k's input copy overlaps step k-1's GEMMs and step k-2's "
                               "result copy (copy streams for each direction, event-ordered)",
                   "ceiling": f"the same host<->device copies without the GEMMs take {c_ms * 1e3:.1f} us per step"}

    extras = [x for x in args.extra_configs.split(",") if x and x != args.config]
    if extras:
        del runner
        torch.cuda.empty_cache()
        line["configs_extra"] = {x: measure_extra(G, x, lut, l2, launch_flag, flush,
                                                  max(2000, args.steps), (hbm, tf_burst, tf_sust))
                                 for x in extras}
        if G.goldy_device_error(clear=True) != 0:
            raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")

    if rank == 0 and not args.no_cpu:
        flops, secs, threads, desc = oracle_sample(st, budget_s=10.0)
        line["cpu_baseline"] = {"value": flops / secs / 1e12, "unit": "TFLOP/s", "cores": threads,
                                "kind": "oracle", "sample": desc + f", {secs:.1f} s"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier(device_ids=[local])
        dist.destroy_process_group()
    return 0


def time_policies(st, lut, copies, steps):
    """Makespan (us) of one set under each policy, timed like the main line
    (each timed region after 0.1 s of its own steps: a GPU left idle while the
    host builds the next set's runs starts below its clocks)."""
    import torch
    from paper_2409_02227_gb300 import goldy as G
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype, batch=s.batch) for s in st.specs]
    out = {}
    predictor = G.goldy_predictor_load() if os.path.exists(G.DEFAULT_PREDICTOR) else None
    for name, flags in (("goldyloc", G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED),
                        ("goldyloc_lr", G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED),
                        ("goldyloc_streams", G.GOLDY_PLAN_AUTO),
                        ("sequential", G.GOLDY_PLAN_SEQUENTIAL),
                        ("naive_streams", G.GOLDY_PLAN_DEFAULT),
                        ("go_all_concurrent", G.GOLDY_PLAN_GO)):
        if name == "goldyloc_lr":
            if predictor is None:
                continue
            sched = G.goldy_plan_ex(descs, lut, predictor, flags)
        else:
            sched = G.goldy_plan(descs, lut, flags)
        out[name], out.setdefault("by_replay", {})[name] = time_schedule(st, sched, copies, steps, soak_s=0.1)
        if name in ("goldyloc", "goldyloc_lr"):
            out["plan" if name == "goldyloc" else "plan_lr"] = [G.goldy_schedule_entry(sched, i)
                                                                 for i in range(len(descs))]
    if G.goldy_device_error(clear=True) != 0:
        raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")
    return out


def run_report(args, local):
    """Every fixed set and the 64 randomized sets under every policy."""
    import torch
    torch.cuda.set_device(local)
    from paper_2409_02227_gb300 import goldy as G
    from paper_2409_02227_gb300 import workloads as wl
    lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    hbm, tf_burst, _, _ = peaks()
    l2 = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 126 * 2 ** 20))
    rows = []
    flush = torch.empty(2 * l2, dtype=torch.uint8, device="cuda")
    sets = [(n, wl.make_config(n)) for n in wl.FIXED_CONFIGS]
    sets += [(f"sweep_{j:02d}", None) for j in range(wl.SWEEP_SETS)]
    for name, st in sets:
        if st is None:
            st = wl.make_sweep_set(int(name.split("_")[1]))
        in_bytes = sum(s.batch * (2 * s.M * s.K + 2 * s.K * s.N) for s in st.specs)
        copies = max(2, math.ceil(2 * l2 / in_bytes))
        steps = max(50, min(2000, int(2e5 / max(1.0, st.flops / 1e9))))
        t = time_policies(st, lut, copies, steps)
        # single steps of the GOLDYLOC plan, each with its own events: L2-cold
        # (flushed) and warm, median and p10 / p90
        descs = [G.desc(s.M, s.N, s.K, s.out_dtype, batch=s.batch) for s in st.specs]
        r = SetRunner(st, G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED), copies)
        step_cold = r.step_distribution(60, "cold", flush)
        step_warm = r.step_distribution(60, "warm")
        del r
        if name in wl.FIXED_CONFIGS:
            cb = cublas_reference_ms(st, copies, steps)
            t["cublas_sequential_reference"] = cb["sequential"] * 1e3
            t["cublas_streams_reference"] = cb["streams"] * 1e3
        roof_us = max(st.flops / (tf_burst * 1e12), st.bytes / (hbm * 1e9)) * 1e6
        row = {"set": name, "n_gemms": len(st.specs), "flops": st.flops, "bytes": st.bytes,
               "bound": "tensor" if st.flops / st.bytes > tf_burst * 1e12 / (hbm * 1e9) else "hbm",
               "roof_us": roof_us,
               "us": {k: v for k, v in t.items() if not k.startswith("plan") and k != "by_replay"},
               "us_by_replay": t["by_replay"],
               "tflops": st.flops / (t["goldyloc"] * 1e-6) / 1e12,
               "roofline_frac": roof_us / t["goldyloc"],
               "speedup_vs_sequential": t["sequential"] / t["goldyloc"],
               "speedup_vs_naive_streams": t["naive_streams"] / t["goldyloc"],
               "plan": [{"group": g, "variant": G.goldy_variant_info_get(v)["name"], "slot": sl, "cd": cd}
                        for g, v, sl, cd in t["plan"]],
               "plan_lr_differs": t.get("plan_lr", t["plan"]) != t["plan"],
               "goldyloc_step_cold_us": step_cold, "goldyloc_step_warm_us": step_warm}
        rows.append(row)
        cb_s = f"{t['cublas_sequential_reference']:.2f} / {t['cublas_streams_reference']:.2f}" \
            if "cublas_streams_reference" in t else ""
        print(f"| {name} | {len(st.specs)} | {row['bound']} | {roof_us:.2f} | {t['goldyloc']:.2f} | "
              f"{row['tflops']:.1f} | {row['roofline_frac']:.3f} | {row['speedup_vs_sequential']:.2f} | "
              f"{row['speedup_vs_naive_streams']:.2f} | {t.get('goldyloc_lr', float('nan')):.2f} | "
              f"{step_cold['median_us']:.2f} ({step_cold['p10_us']:.2f}-{step_cold['p90_us']:.2f}) | "
              f"{step_warm['median_us']:.2f} ({step_warm['p10_us']:.2f}-{step_warm['p90_us']:.2f}) | {cb_s} |",
              flush=True)
        del st
        torch.cuda.empty_cache()
    sweep = [r for r in rows if r["set"].startswith("sweep")]
    geo = lambda xs: math.exp(sum(math.log(x) for x in xs) / len(xs))
    lr_rows = [r for r in sweep if "goldyloc_lr" in r["us"]]
    summary = {"sweep_geomean_speedup_vs_sequential": geo([r["speedup_vs_sequential"] for r in sweep]),
               "sweep_geomean_speedup_vs_naive_streams": geo([r["speedup_vs_naive_streams"] for r in sweep]),
               "sweep_geomean_roofline_frac": geo([r["roofline_frac"] for r in sweep]),
               "sweep_geomean_roofline_frac_tensor_bound": geo([r["roofline_frac"] for r in sweep
                                                                if r["bound"] == "tensor"] or [1.0]),
               "sweep_sets_faster_than_sequential": sum(r["speedup_vs_sequential"] > 1 for r in sweep),
               "sweep_sets_faster_than_naive_streams": sum(r["speedup_vs_naive_streams"] > 1 for r in sweep)}
    if lr_rows:
        # the predictor-planned schedule against the table-planned one (Sec. 4.3)
        summary["sweep_geomean_lr_over_table_time"] = geo([r["us"]["goldyloc_lr"] / r["us"]["goldyloc"]
                                                           for r in lr_rows])
        summary["sweep_geomean_lr_speedup_vs_sequential"] = geo([r["us"]["sequential"] / r["us"]["goldyloc_lr"]
                                                                 for r in lr_rows])
        summary["sweep_sets_lr_plan_differs"] = sum(r.get("plan_lr_differs", False) for r in lr_rows)
    print(json.dumps(summary), flush=True)
    with open(args.report, "w") as f:
        json.dump({"rows": rows, "summary": summary, "peaks": {"hbm_gbs": hbm, "bf16_tflops": tf_burst}}, f, indent=1)
    return 0


TRACE_PHASES = (  # (slot, name) of goldy_run_opts.trace, in the order they happen
    (0, "CTA start"), (10, "set-up done (before the dependency wait)"), (11, "producer starts"),
    (2, "first stage's loads issued"), (3, "first stage landed (MMA thread)"),
    (1, "epilogue past the dependency wait"), (4, "first accumulator committed"),
    (5, "first accumulator seen by the epilogue"), (6, "split-K partial staged / sent"),
    (7, "split-K partials received / arrival counted"), (8, "first unit stored"), (9, "CTA done"))


def run_phase_trace(args, local):
    """One step of the planned set traced on the device (%globaltimer stamps
    per CTA, goldy_run_opts.trace) while it runs among back-to-back steps the
    way the bench line replays them; per launch, the median and p90 over its
    CTAs of each phase, in us from the step's first CTA start."""
    import numpy as np
    import torch
    torch.cuda.set_device(local)
    from paper_2409_02227_gb300 import goldy as G
    st = load_set(args.config)
    lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    launch_flag = G.GOLDY_PLAN_FUSED if args.launch == "fused" else 0
    descs, sched, plan, single = plan_set(G, st, lut, launch_flag)
    l2 = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 126 * 2 ** 20))
    copies, _ = rotating_copies(st, l2)
    ready = not args.no_inputs_ready
    r = SetRunner(st, sched, copies, serial_launch=args.serial_launch, inputs_ready=ready)
    us = r.timed(200) / 200 * 1e3
    cta_cap = 1 << 16
    tr = torch.zeros(cta_cap * 16, dtype=torch.int64, device="cuda")
    A, B, C = r.copies[0]
    ex = G.goldy_exec_create(sched, [a.data_ptr() for a in A], [b.data_ptr() for b in B], [c.data_ptr() for c in C],
                             r.ws.data_ptr(), r.ws_bytes, [x.cuda_stream for x in r.streams], trace=tr.data_ptr(),
                             trace_ctas=cta_cap, serial_launch=args.serial_launch, inputs_ready=ready)
    r.spin(200)
    for k in range(1, 12):             # copies 1.., the traced step (copy 0) in the middle
        r.launch(k if k % copies else k + 1)
        if k == 6:
            G.goldy_exec_launch(ex)
    torch.cuda.synchronize()
    if G.goldy_device_error(clear=True) != 0:
        raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")
    a = tr.view(cta_cap, 16).cpu().numpy().astype(np.int64)
    launches, off = [], 0
    while off < cta_cap and a[off, 12] > 0:
        g = int(a[off, 12])
        launches.append(a[off:off + g])
        off += g
    t0 = min(int(l[:, 0].min()) for l in launches)
    names = [G.goldy_variant_info_get(v)["name"] for _, v, _, _ in plan]
    print(f"# Phase trace: {args.config} ({workload_label(st.specs)})\n")
    print(f"Plan: {', '.join(sorted(set(names)))}; {len(launches)} launch(es) per step; "
          f"back-to-back step time {us:.2f} us ({'inputs_ready' if ready else 'no inputs_ready'}).\n")
    for j, l in enumerate(launches):
        print(f"Launch {j}: grid {len(l)} CTAs, {int(l[:, 14].sum())} units, SMs used {len(set(l[:, 15].tolist()))}\n")
        print("| phase | median us | p90 us |")
        print("|---|---|---|")
        for slot, name in TRACE_PHASES:
            v = l[:, slot]
            v = v[v > 0]
            if v.size == 0:
                continue
            x = (v - t0) / 1e3
            print(f"| {name} | {np.median(x):.2f} | {np.percentile(x, 90):.2f} |")
        print()
    return 0


SCALING_PARTITIONS = ((38, "GPU-Quarter"), (76, "GPU-Half"), (0, "GPU"))


def scaling_lut_path(sm_count: int) -> str:
    from paper_2409_02227_gb300 import goldy as G
    return os.path.join(os.path.dirname(G.DEFAULT_LUT), "scaling", f"goldy_lut_sm{sm_count}.bin")


def run_scaling_study(args, local):
    """GPU-scaling study (Sec. 7.4, Scaling GPUs Configuration): each study set (4 equal GEMMs, CD 4) run
    inside SM partitions of a quarter, half and all of the GPU, under the
    default configuration (isolation-tuned kernels, all GEMMs on their own
    streams), sequential, GOLDYLOC with the table tuned inside that partition,
    and GOLDYLOC re-using the whole-GPU table.  Everything is timed inside the
    partition (prepared runs, events in the partition)."""
    import torch
    torch.cuda.set_device(local)
    from paper_2409_02227_gb300 import goldy as G
    from paper_2409_02227_gb300 import workloads as wl
    l2 = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 126 * 2 ** 20))
    full_lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    n_sets = len(wl.scaling_study_shapes())
    rows, summary = [], {}
    geo = lambda xs: math.exp(sum(math.log(x) for x in xs) / len(xs))
    for req, label in SCALING_PARTITIONS:
        part = G.goldy_partition_create(req, 16)
        sm, streams = G.goldy_partition_query(part, 16)
        path = scaling_lut_path(sm)
        tuned = G.goldy_lut_load(path) if os.path.exists(path) else None
        for i in range(n_sets):
            st = wl.make_scaling_set(i)
            descs = [G.desc(x.M, x.N, x.K, x.out_dtype) for x in st.specs]
            in_bytes = sum(2 * x.M * x.K + 2 * x.K * x.N for x in st.specs)
            copies = min(16, max(2, math.ceil(2 * l2 / in_bytes)))
            base_a = [a.cuda() for a in st.a]
            base_b = [b.cuda() for b in st.b]
            cdt = [torch.bfloat16 if x.out_dtype == 0 else torch.float32 for x in st.specs]
            bufs = []
            for r in range(copies):
                A = base_a if r == 0 else [a.clone() for a in base_a]
                B = base_b if r == 0 else [b.clone() for b in base_b]
                C = [torch.empty((x.M, x.N), dtype=d, device="cuda") for x, d in zip(st.specs, cdt)]
                bufs.append((A, B, C))
            torch.cuda.synchronize()
            pols = [("default", full_lut if tuned is None else tuned, G.GOLDY_PLAN_DEFAULT),
                    ("sequential", full_lut if tuned is None else tuned, G.GOLDY_PLAN_SEQUENTIAL),
                    ("goldyloc_whole_gpu_table", full_lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)]
            if tuned is not None:
                pols.append(("goldyloc", tuned, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED))
            us = {}
            for name, lut, flags in pols:
                sched = G.goldy_plan(descs, lut, flags)
                _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
                ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
                torch.cuda.synchronize()
                execs = [G.goldy_exec_create(sched, [a.data_ptr() for a in A], [b.data_ptr() for b in B],
                                             [c.data_ptr() for c in C], ws.data_ptr(), ws_bytes,
                                             streams[:max(1, ms)]) for A, B, C in bufs]
                est = G.goldy_exec_time(execs, 2 * copies, copies) * 1e3
                reps = int(min(2000, max(3 * copies, 20000.0 / max(est, 1.0))))
                us[name] = G.goldy_exec_time(execs, 0, reps) * 1e3
                del execs, ws
            if G.goldy_device_error(clear=True) != 0:
                raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")
            x = st.specs[0]
            row = {"partition": label, "sms": sm, "set": st.name, "gemm": [x.M, x.N, x.K, x.out_dtype],
                   "us": us}
            rows.append(row)
            del bufs, base_a, base_b, st
            torch.cuda.empty_cache()
        mine = [r for r in rows if r["partition"] == label]
        best = "goldyloc" if tuned is not None else "goldyloc_whole_gpu_table"
        summary[label] = {
            "sms": sm, "table": path if tuned is not None else "whole-GPU table (no partition table found)",
            "geomean_speedup_vs_default": geo([r["us"]["default"] / r["us"][best] for r in mine]),
            "geomean_speedup_vs_sequential": geo([r["us"]["sequential"] / r["us"][best] for r in mine]),
            "geomean_speedup_whole_gpu_table_vs_default": geo([r["us"]["default"] / r["us"]["goldyloc_whole_gpu_table"]
                                                               for r in mine]),
            "sets_faster_than_default": sum(r["us"]["default"] > r["us"][best] for r in mine), "sets": len(mine)}
        print(label, json.dumps(summary[label]), flush=True)
        del part
    with open(args.scaling_study, "w") as f:
        json.dump({"rows": rows, "summary": summary}, f, indent=1)
    return 0


def run_batched_study(args, local):
    """Heterogeneous strided-batched GEMMs (Sec. 6.7): sets of 2 and 4
    batched attention GEMMs over variable sequence lengths, under default
    (isolation-tuned kernels, every B-GEMM on its own stream), sequential,
    GO at CD = n, and GOLDYLOC; each configuration at its faster replay,
    inputs rotated past the L2."""
    import torch
    torch.cuda.set_device(local)
    from paper_2409_02227_gb300 import goldy as G
    from paper_2409_02227_gb300 import workloads as wl
    l2 = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 126 * 2 ** 20))
    lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    rows = []
    for members in (2, 4):
        for i in range(16):
            st = wl.make_batched_set(i, members)
            descs = [G.desc(x.M, x.N, x.K, x.out_dtype, batch=x.batch) for x in st.specs]
            in_bytes = sum(x.batch * (2 * x.M * x.K + 2 * x.K * x.N) for x in st.specs)
            copies = min(16, max(2, math.ceil(2 * l2 / in_bytes)))
            steps = max(50, min(2000, int(2e5 / max(1.0, st.flops / 1e9))))
            us, plans = {}, {}
            for name, flags in (("default", G.GOLDY_PLAN_DEFAULT), ("sequential", G.GOLDY_PLAN_SEQUENTIAL),
                                ("go_all_concurrent", G.GOLDY_PLAN_GO | G.GOLDY_PLAN_FUSED),
                                ("goldyloc", G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)):
                sched = G.goldy_plan(descs, lut, flags)
                us[name], _ = time_schedule(st, sched, copies, steps)
                plans[name] = [G.goldy_schedule_entry(sched, k) for k in range(len(descs))]
            if G.goldy_device_error(clear=True) != 0:
                raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")
            rows.append({"set": st.name, "members": members,
                         "gemms": [[x.M, x.N, x.K, x.batch] for x in st.specs], "us": us,
                         "goldyloc_plan": [{"group": g, "variant": G.goldy_variant_info_get(v)["name"], "cd": cd}
                                           for g, v, _, cd in plans["goldyloc"]]})
            print(st.name, {k: round(v, 2) for k, v in us.items()}, flush=True)
            del st
            torch.cuda.empty_cache()
    geo = lambda xs: math.exp(sum(math.log(x) for x in xs) / len(xs))
    summary = {}
    for members in (2, 4):
        sel = [r for r in rows if r["members"] == members]
        summary[f"{members}P"] = {
            "sets": len(sel),
            "goldyloc_speedup_vs_default": geo([r["us"]["default"] / r["us"]["goldyloc"] for r in sel]),
            "goldyloc_max_speedup_vs_default": max(r["us"]["default"] / r["us"]["goldyloc"] for r in sel),
            "goldyloc_speedup_vs_sequential": geo([r["us"]["sequential"] / r["us"]["goldyloc"] for r in sel]),
            "go_speedup_vs_default": geo([r["us"]["default"] / r["us"]["go_all_concurrent"] for r in sel])}
    print(json.dumps(summary), flush=True)
    with open(args.batched_study, "w") as f:
        json.dump({"rows": rows, "summary": summary}, f, indent=1)
    return 0


def run_corun_study(args, local):
    """GEMM + element-wise add (Sec. 7.1): each study GEMM co-scheduled with
    an add over its output size under sequential, default (isolation-tuned
    GEMM kernel and the add at once), GO (CD-2 GO-Kernel and a half-GPU add at
    once) and GOLDYLOC (GO where the table marks co-running as paying, else
    sequential).  Prepared runs, inputs rotated past the L2."""
    import torch
    torch.cuda.set_device(local)
    from paper_2409_02227_gb300 import goldy as G
    from paper_2409_02227_gb300 import workloads as wl
    l2 = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 126 * 2 ** 20))
    hbm, tf_burst, _, _ = peaks()
    ridge = tf_burst * 1e12 / (hbm * 1e9)
    lut = G.goldy_lut_load(args.lut or G.DEFAULT_LUT)
    streams = [torch.cuda.Stream() for _ in range(2)]
    sp = [x.cuda_stream for x in streams]
    rows = []
    for i, (M, N, K, out) in enumerate(wl.scaling_study_shapes()):
        td = torch.bfloat16 if out == G.GOLDY_BF16 else torch.float32
        es = 2 if out == G.GOLDY_BF16 else 4
        in_bytes = 2 * M * K + 2 * K * N + 2 * es * M * N
        copies = min(16, max(2, math.ceil(2 * l2 / in_bytes)))
        g = torch.Generator(device="cuda")
        g.manual_seed(4000 + i)
        bufs = []
        for _ in range(copies):
            bufs.append(((torch.rand((M, K), generator=g, device="cuda") - 0.5).to(torch.bfloat16),
                         (torch.rand((K, N), generator=g, device="cuda") - 0.5).to(torch.bfloat16),
                         torch.empty((M, N), dtype=td, device="cuda"),
                         torch.randn(M * N, generator=g, device="cuda").to(td),
                         torch.randn(M * N, generator=g, device="cuda").to(td),
                         torch.empty(M * N, dtype=td, device="cuda")))
        us, plan = {}, {}
        for name, pol in (("sequential", G.GOLDY_PLAN_SEQUENTIAL), ("default", G.GOLDY_PLAN_DEFAULT),
                          ("go", G.GOLDY_PLAN_GO), ("goldyloc", G.GOLDY_PLAN_AUTO)):
            c = G.goldy_corun_plan(G.desc(M, N, K, out), M * N, out, lut, pol)
            conc, v, rc, ws_bytes = G.goldy_corun_query(c)
            ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
            torch.cuda.synchronize()
            execs = [G.goldy_corun_exec_create(c, A.data_ptr(), B.data_ptr(), C.data_ptr(), ws.data_ptr(), ws_bytes,
                                               X.data_ptr(), Y.data_ptr(), Z.data_ptr(), sp)
                     for A, B, C, X, Y, Z in bufs]
            est = G.goldy_exec_time(execs, 2 * copies, copies) * 1e3
            reps = int(min(4000, max(3 * copies, 20000.0 / max(est, 1.0))))
            us[name] = G.goldy_exec_time(execs, 0, reps) * 1e3
            plan[name] = {"concurrent": conc, "variant": G.goldy_variant_info_get(v)["name"], "add_rc_div": rc}
            del execs, ws
        if G.goldy_device_error(clear=True) != 0:
            raise RuntimeError("a GO-Kernel reported a bounded-wait timeout")
        flops = 2 * M * N * K
        gemm_bytes = 2 * M * K + 2 * K * N + es * M * N
        rows.append({"gemm": [M, N, K, out], "memory_bound_gemm": flops / gemm_bytes < ridge, "us": us,
                     "plan": plan})
        del bufs
        torch.cuda.empty_cache()
    geo = lambda xs: math.exp(sum(math.log(x) for x in xs) / len(xs)) if xs else None
    summary = {}
    for sub, sel in (("all", rows), ("memory_bound", [r for r in rows if r["memory_bound_gemm"]]),
                     ("compute_bound", [r for r in rows if not r["memory_bound_gemm"]])):
        summary[sub] = {"gemms": len(sel)}
        for name in ("sequential", "go", "goldyloc"):
            summary[sub][f"{name}_speedup_vs_default"] = geo([r["us"]["default"] / r["us"][name] for r in sel])
        summary[sub]["goldyloc_co_runs"] = sum(r["plan"]["goldyloc"]["concurrent"] for r in sel)
    print(json.dumps(summary), flush=True)
    with open(args.corun_study, "w") as f:
        json.dump({"rows": rows, "summary": summary}, f, indent=1)
    return 0


def main(argv=None):
    args = parse_args(argv)
    world, rank, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, world, rank)
    if args.report:
        return run_report(args, local)
    if args.phase_trace:
        return run_phase_trace(args, local)
    if args.scaling_study:
        return run_scaling_study(args, local)
    if args.corun_study:
        return run_corun_study(args, local)
    if args.batched_study:
        return run_batched_study(args, local)
    return run_gpu(args, world, rank, local)


if __name__ == "__main__":
    sys.exit(main())

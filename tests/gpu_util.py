"""Helpers for the GPU tests: put seeded inputs on the device, run a schedule
through the C ABI, bring results back, compare with the oracle."""
from __future__ import annotations

import numpy as np
import torch

from oracle import gemm as og
from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl

TORCH_OUT = {G.GOLDY_F32: torch.float32, G.GOLDY_BF16: torch.bfloat16}


class Launch:
    """Device buffers + streams for one schedule over one set of inputs."""

    def __init__(self, sched, As, Bs, out_dtypes, fill=float("nan")):
        self.sched = sched
        n, _, max_streams, ws_bytes = G.goldy_schedule_query(sched)
        self.ws_bytes = ws_bytes
        self.dA = [a.cuda() for a in As]
        self.dB = [b.cuda() for b in Bs]
        self.dC = [torch.full((a.shape[0], b.shape[1]), fill, dtype=TORCH_OUT[o], device="cuda")
                   for a, b, o in zip(As, Bs, out_dtypes)]
        self.ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
        self.streams = [torch.cuda.Stream() for _ in range(max(1, max_streams))]

    def ptrs(self):
        return ([a.data_ptr() for a in self.dA], [b.data_ptr() for b in self.dB],
                [c.data_ptr() for c in self.dC])

    def run(self):
        A, B, C = self.ptrs()
        self.streams[0].wait_stream(torch.cuda.current_stream())
        G.goldy_run(self.sched, A, B, C, self.ws.data_ptr(), self.ws_bytes,
                    [s.cuda_stream for s in self.streams])
        torch.cuda.current_stream().wait_stream(self.streams[0])

    def graph(self):
        A, B, C = self.ptrs()
        torch.cuda.synchronize()
        return G.goldy_graph_create(self.sched, A, B, C, self.ws.data_ptr(), self.ws_bytes,
                                    [s.cuda_stream for s in self.streams])

    def exec(self):
        A, B, C = self.ptrs()
        return G.goldy_exec_create(self.sched, A, B, C, self.ws.data_ptr(), self.ws_bytes,
                                   [s.cuda_stream for s in self.streams])

    def results(self):
        torch.cuda.synchronize()
        err = G.goldy_device_error(clear=True)
        assert err == 0, f"kernel reported error word {err}"
        return [c.cpu() for c in self.dC]


def run_explicit(As, Bs, out_dtypes, variants, groups=None, slots=None):
    n = len(As)
    descs = [G.desc(a.shape[0], b.shape[1], a.shape[1], o) for a, b, o in zip(As, Bs, out_dtypes)]
    s = G.goldy_schedule_build(descs, groups or [0] * n, variants, slots or list(range(n)))
    L = Launch(s, As, Bs, out_dtypes)
    L.run()
    return L.results()


def check_close(got: torch.Tensor, a: torch.Tensor, b: torch.Tensor, label=""):
    """|gpu - ref| <= 1e-2 * max|ref| + 1e-3 elementwise against the fp64 oracle."""
    ref = og.gemm(wl.bits_of(a), wl.bits_of(b))
    g = got.to(torch.float64).numpy()
    assert np.all(np.isfinite(g)), f"{label}: non-finite output (unwritten elements?)"
    tol = og.tolerance(ref)
    err = np.abs(g - ref)
    worst = float(err.max()) if err.size else 0.0
    assert worst <= tol, f"{label}: max |gpu-ref| = {worst:.3e} > tol {tol:.3e}"
    return worst, tol


def check_rows(got: torch.Tensor, a: torch.Tensor, b: torch.Tensor, rows, label=""):
    """Same bar on a sample of rows (each computed exactly by the oracle);
    max|ref| is taken over the sampled rows."""
    ref = og.gemm_rows(wl.bits_of(a), wl.bits_of(b), rows)
    g = got[torch.as_tensor(rows)].to(torch.float64).numpy()
    assert np.all(np.isfinite(g)), f"{label}: non-finite output"
    tol = og.tolerance(ref)
    worst = float(np.abs(g - ref).max())
    assert worst <= tol, f"{label}: max |gpu-ref| = {worst:.3e} > tol {tol:.3e}"
    return worst, tol

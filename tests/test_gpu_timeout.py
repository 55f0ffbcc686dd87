"""The bounded-wait timeout path, exercised on the GPU without a fault.

The run option ``test_stall_first_stage`` makes CTA 0 of the run's first
GO-Kernel launch leave its first shared-memory stage unfilled: no copy is
issued and no address is touched, so the MMA thread's bounded wait for that
stage runs out (here after 2 ms, ``wait_limit_us``).  The kernel must then
return by itself, the error word must read 2 (an MMA-thread wait gave up),
and the next normal run must match the oracle — after the workspace is
zero-filled again, as the header asks for after a device error (the stalled
split never arrived, so a split-K arrival counter was left non-zero)."""
import numpy as np
import pytest
import torch

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import check_close

pytestmark = pytest.mark.gpu

F32 = G.GOLDY_F32
KIND_N128_FULL = 2
WAIT_US = 2000
ERR_MMA_WAIT = 2


def _setup(shapes, variants, flags):
    As = [wl.random_matrix(M, K, 90 + i, "normal", 0.1) for i, (M, N, K) in enumerate(shapes)]
    Bs = [wl.random_matrix(K, N, 95 + i, "normal", 0.1) for i, (M, N, K) in enumerate(shapes)]
    descs = [G.desc(M, N, K, F32) for M, N, K in shapes]
    n = len(shapes)
    s = G.goldy_schedule_build(descs, [0] * n, variants, list(range(n)), flags)
    _, _, ms, ws_bytes = G.goldy_schedule_query(s)
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    dA = [a.cuda() for a in As]
    dB = [b.cuda() for b in Bs]
    dC = [torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda") for M, N, K in shapes]
    streams = [torch.cuda.Stream() for _ in range(max(1, ms))]
    return As, Bs, s, ws, ws_bytes, dA, dB, dC, streams


def _run(s, ws, ws_bytes, dA, dB, dC, streams, **opts):
    streams[0].wait_stream(torch.cuda.current_stream())
    G.goldy_run_ex(s, [a.data_ptr() for a in dA], [b.data_ptr() for b in dB], [c.data_ptr() for c in dC],
                   ws.data_ptr(), ws_bytes, [x.cuda_stream for x in streams], **opts)
    torch.cuda.current_stream().wait_stream(streams[0])
    torch.cuda.synchronize()


def test_stalled_stage_times_out_and_the_kernel_returns(cuda_ok):
    assert G.goldy_device_error(clear=True) == 0
    shapes = [(512, 512, 1024)]
    As, Bs, s, ws, ws_bytes, dA, dB, dC, streams = _setup(shapes, [G.variant_id(KIND_N128_FULL, 1, 1)], 0)
    _run(s, ws, ws_bytes, dA, dB, dC, streams, wait_limit_us=WAIT_US, test_stall_first_stage=True)
    assert G.goldy_device_error(clear=True) == ERR_MMA_WAIT
    # CTA 0's first unit (the tile at rows 0..127, columns 0..127) was never computed
    assert torch.isnan(dC[0][:128, :128].cpu()).all()
    # the context is still usable: a normal run gives the oracle's result
    dC[0].fill_(float("nan"))
    _run(s, ws, ws_bytes, dA, dB, dC, streams)
    assert G.goldy_device_error(clear=True) == 0
    check_close(dC[0].cpu(), As[0], Bs[0], "after a timed-out run")


def test_workspace_zeroed_again_after_a_timeout_recovers(cuda_ok):
    # two GEMMs of one kind with different K splits in one fused launch: the
    # splits of a tile meet through arrival counters in the workspace (the
    # last to arrive sums them)
    assert G.goldy_device_error(clear=True) == 0
    shapes = [(256, 512, 1024), (256, 512, 1024)]
    vs = [G.variant_id(KIND_N128_FULL, 2, 1), G.variant_id(KIND_N128_FULL, 4, 1)]
    As, Bs, s, ws, ws_bytes, dA, dB, dC, streams = _setup(shapes, vs, G.GOLDY_PLAN_FUSED)
    assert ws_bytes > 0
    _run(s, ws, ws_bytes, dA, dB, dC, streams, wait_limit_us=WAIT_US, test_stall_first_stage=True)
    assert G.goldy_device_error(clear=True) == ERR_MMA_WAIT
    ws.zero_()
    for c in dC:
        c.fill_(float("nan"))
    for _ in range(2):
        _run(s, ws, ws_bytes, dA, dB, dC, streams)
        assert G.goldy_device_error(clear=True) == 0
        for i in range(2):
            check_close(dC[i].cpu(), As[i], Bs[i], f"gemm {i} after the workspace was zeroed again")

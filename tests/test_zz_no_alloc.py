"""goldy_gemm_noalloc: one GEMM for callers that may not allocate device
memory (fixed-budget runtimes, frameworks that own every device allocation,
paths that cannot afford cudaMalloc's implicit synchronisation).  Its split-K
scratch is a fixed array inside the library.

The GPU test runs the same GEMM and variant through goldy_run (caller
workspace) and then twice in a row through goldy_gemm_noalloc on one stream;
both calls must agree with goldy_run within the parity bar
|x - y| <= 1e-2 * max|ref| + 1e-3 (they are in fact byte-identical: the same
kernel sums every element in the same order), and with the fp64 oracle at the
same bar.  A second case runs both entry points on the streams of an SM
partition.  This file sorts last so that a run stopping at its first failure
has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import check_close

F32, BF16 = G.GOLDY_F32, G.GOLDY_BF16
TORCH_OUT = {F32: torch.float32, BF16: torch.bfloat16}

CASES = [
    # M, N, K, out, kind, split
    (128, 1024, 4096, BF16, 1, 4),    # 128x64 tiles, two CTAs per SM, split 4
    (32, 4096, 1024, F32, 7, 2),      # transposed 32x128 tiles, split 2
    (200, 320, 448, F32, 3, 8),       # ragged tails; split 8 is clamped to the 7 K blocks
]


@pytest.mark.gpu
@pytest.mark.parametrize("M,N,K,out,kind,split", CASES)
def test_noalloc_matches_goldy_run_twice(cuda_ok, M, N, K, out, kind, split):
    a = wl.random_matrix(M, K, seed=70 + M, dist="normal", scale=0.5)
    b = wl.random_matrix(K, N, seed=71 + N, dist="normal", scale=0.5)
    v = G.variant_id(kind, split, 1)
    d = G.desc(M, N, K, out)
    dA, dB = a.cuda(), b.cuda()
    stream = torch.cuda.current_stream()

    # the existing entry point, with a caller-allocated workspace
    sched = G.goldy_schedule_build([d], [0], [v], [0])
    _, _, _, ws_bytes = G.goldy_schedule_query(sched)
    assert ws_bytes > 0                    # the variant really uses scratch memory
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    ref = torch.full((M, N), float("nan"), dtype=TORCH_OUT[out], device="cuda")
    G.goldy_run(sched, [dA.data_ptr()], [dB.data_ptr()], [ref.data_ptr()], ws.data_ptr(), ws_bytes,
                [stream.cuda_stream])

    outs = []
    for _ in range(2):                     # two calls in a row share the static scratch
        c = torch.full((M, N), float("nan"), dtype=TORCH_OUT[out], device="cuda")
        G.goldy_gemm_noalloc(d, v, dA.data_ptr(), dB.data_ptr(), c.data_ptr(), stream.cuda_stream)
        outs.append(c)
    torch.cuda.synchronize()
    assert G.goldy_device_error(clear=True) == 0

    r = ref.cpu().double().numpy()
    assert np.all(np.isfinite(r))
    tol = 1e-2 * float(np.abs(r).max()) + 1e-3
    for c in outs:
        x = c.cpu().double().numpy()
        assert np.all(np.isfinite(x))
        assert float(np.abs(x - r).max()) <= tol
        assert torch.equal(c.cpu().view(torch.uint8), ref.cpu().view(torch.uint8))
        check_close(c.cpu(), a, b, f"noalloc {M}x{N}x{K} kind {kind} split {split}")


def _stream_sync(handle):
    """cuStreamSynchronize on a driver stream handle (a partition's stream
    lives in its green context, which a device-wide synchronise of the
    primary context does not cover)."""
    rc = ctypes.CDLL("libcuda.so.1").cuStreamSynchronize(ctypes.c_void_p(handle))
    assert rc == 0, f"cuStreamSynchronize returned {rc}"


@pytest.mark.gpu
def test_noalloc_inside_a_partition_matches_goldy_run(cuda_ok):
    """On a partition's stream the entry point runs inside the partition: the
    same grid caps as goldy_run there, so the same bytes."""
    M, N, K, out, kind, split = 128, 1024, 4096, BF16, 1, 4
    a = wl.random_matrix(M, K, seed=80, dist="normal", scale=0.5)
    b = wl.random_matrix(K, N, seed=81, dist="normal", scale=0.5)
    v = G.variant_id(kind, split, 1)
    d = G.desc(M, N, K, out)
    dA, dB = a.cuda(), b.cuda()
    part = G.goldy_partition_create(38, 2)
    sms, streams = G.goldy_partition_query(part, 1)
    assert sms < torch.cuda.get_device_properties(0).multi_processor_count
    sched = G.goldy_schedule_build([d], [0], [v], [0])
    _, _, _, ws_bytes = G.goldy_schedule_query(sched)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    ref = torch.full((M, N), float("nan"), dtype=TORCH_OUT[out], device="cuda")
    outs = [torch.full((M, N), float("nan"), dtype=TORCH_OUT[out], device="cuda") for _ in range(2)]
    torch.cuda.synchronize()
    G.goldy_run(sched, [dA.data_ptr()], [dB.data_ptr()], [ref.data_ptr()], ws.data_ptr(), ws_bytes, streams)
    for c in outs:
        G.goldy_gemm_noalloc(d, v, dA.data_ptr(), dB.data_ptr(), c.data_ptr(), streams[0])
    _stream_sync(streams[0])
    assert G.goldy_device_error(clear=True) == 0
    for c in outs:
        assert torch.equal(c.cpu().view(torch.uint8), ref.cpu().view(torch.uint8))
        check_close(c.cpu(), a, b, "noalloc in a partition")
    del part


def test_noalloc_rejects_requests_beyond_its_scratch():
    # 2048 x 8192 with 128x256 tiles split 8: 512 tiles x 8 x 128 KiB of partials
    d = G.desc(2048, 8192, 2048, F32)
    with pytest.raises(G.GoldyError) as e:
        G.goldy_gemm_noalloc(d, G.variant_id(4, 8, 1), 16, 16, 16, 0)
    assert e.value.status == G.GOLDY_ERR_INVALID_ARG
    assert "static scratch holds 33554432 bytes" in str(e.value)

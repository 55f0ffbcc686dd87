"""A GEMM co-scheduled with an element-wise add (Sec. 7.1) on the GPU: under
every policy the GEMM matches the oracle and the add matches the oracle bit
for bit (both take the same IEEE fp32 addition and bf16 rounding), over
ragged lengths, unaligned operands (scalar path), n = 0, and through a
prepared run."""
import numpy as np
import pytest
import torch

from oracle import ewise as ew
from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import check_close, check_rows

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _ref_add(x, y, dtype):
    if dtype == G.GOLDY_BF16:
        return ew.add_bf16(_bits(x), _bits(y))
    return ew.add_f32(x.cpu().numpy(), y.cpu().numpy())


def _same(z, ref, dtype):
    got = _bits(z) if dtype == G.GOLDY_BF16 else z.cpu().numpy()
    if dtype == G.GOLDY_BF16:
        return np.array_equal(got, ref)
    return np.array_equal(got.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("dtype", [G.GOLDY_BF16, G.GOLDY_F32])
@pytest.mark.parametrize("n,offset", [(1 << 20, 0), (1000003, 0), (77777, 1), (7, 0), (0, 0)])
def test_ewise_add_bit_exact(cuda_ok, dtype, n, offset):
    g = torch.Generator().manual_seed(n + offset)
    td = torch.bfloat16 if dtype == G.GOLDY_BF16 else torch.float32
    x = (torch.randn(n + offset, generator=g) * 3).to(td).cuda()[offset:]
    y = (torch.randn(n + offset, generator=g) * 0.01).to(td).cuda()[offset:]
    z = torch.full((n + offset,), float("nan"), dtype=td, device="cuda")[offset:]
    for rc in (1, 2, 4):
        s = torch.cuda.current_stream()
        G.goldy_ewise_add(x.data_ptr(), y.data_ptr(), z.data_ptr(), n, dtype, rc, s.cuda_stream)
        torch.cuda.synchronize()
        assert _same(z, _ref_add(x, y, dtype), dtype)


@pytest.mark.parametrize("policy", [G.GOLDY_PLAN_SEQUENTIAL, G.GOLDY_PLAN_DEFAULT, G.GOLDY_PLAN_GO,
                                    G.GOLDY_PLAN_AUTO])
@pytest.mark.parametrize("shape", [(128, 1024, 4096, 0), (512, 1024, 1024, 1), (40, 296, 320, 1)])
def test_corun_results(cuda_ok, policy, shape):
    M, N, K, out = shape
    a = wl.random_matrix(M, K, 11, "normal", 0.05)
    b = wl.random_matrix(K, N, 12, "normal", 0.05)
    lut = G.goldy_lut_load()
    c = G.goldy_corun_plan(G.desc(M, N, K, out), M * N, out, lut, policy)
    conc, v, rc, ws_bytes = G.goldy_corun_query(c)
    td = torch.bfloat16 if out == G.GOLDY_BF16 else torch.float32
    dA, dB = a.cuda(), b.cuda()
    dC = torch.full((M, N), float("nan"), dtype=td, device="cuda")
    gen = torch.Generator().manual_seed(5)
    X = torch.randn(M * N, generator=gen).to(td).cuda()
    Y = torch.randn(M * N, generator=gen).to(td).cuda()
    Z = torch.full((M * N,), float("nan"), dtype=td, device="cuda")
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    streams[0].wait_stream(torch.cuda.current_stream())
    G.goldy_corun_run(c, dA.data_ptr(), dB.data_ptr(), dC.data_ptr(), ws.data_ptr(), ws_bytes, X.data_ptr(),
                      Y.data_ptr(), Z.data_ptr(), [s.cuda_stream for s in streams])
    torch.cuda.current_stream().wait_stream(streams[0])
    torch.cuda.synchronize()
    assert G.goldy_device_error(clear=True) == 0
    check_close(dC.cpu(), a, b, f"corun gemm {shape} policy {policy}")
    ref = _ref_add(X, Y, out)
    assert _same(Z, ref, out)
    # the same co-run as a prepared run, replayed twice
    dC.fill_(float("nan"))
    Z.fill_(float("nan"))
    torch.cuda.synchronize()
    x = G.goldy_corun_exec_create(c, dA.data_ptr(), dB.data_ptr(), dC.data_ptr(), ws.data_ptr(), ws_bytes,
                                  X.data_ptr(), Y.data_ptr(), Z.data_ptr(), [s.cuda_stream for s in streams])
    G.goldy_exec_time([x], 1, 1)
    assert _same(Z, ref, out)
    check_close(dC.cpu(), a, b, f"corun exec gemm {shape} policy {policy}")
    del x

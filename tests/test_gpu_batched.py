"""Strided-batched GEMMs (Sec. 6.7's B-GEMMs) on the GPU: every entry of a
batch matches the oracle under every kernel kind, with split-K (cluster and
last-arriver reductions), fused launches mixing batched and plain GEMMs,
non-packed strides (the gaps between entries stay untouched), K = 0, and
the planner on the batched attention study sets."""
import numpy as np
import pytest
import torch

from oracle import gemm as og
from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import TORCH_OUT, check_close, check_rows

pytestmark = pytest.mark.gpu
F32, BF16 = G.GOLDY_F32, G.GOLDY_BF16
SWAP_KINDS = {6, 7, 8, 9}


def vid(kind, split=1, rc=1):
    return G.variant_id(kind, split, rc)


def batched_inputs(batch, M, N, K, seed):
    a = torch.stack([wl.random_matrix(M, K, seed + 2 * i, "normal", 0.05) for i in range(batch)])
    b = torch.stack([wl.random_matrix(K, N, seed + 2 * i + 1, "normal", 0.05) for i in range(batch)])
    return a, b


def run(descs, As, Bs, outs, variants, groups=None, slots=None, flags=0, c_elems=None, fill=float("nan")):
    """Run an explicit schedule; A/B given as device-ready CPU tensors laid
    out at the descriptors' strides; returns the raw C buffers."""
    n = len(descs)
    s = G.goldy_schedule_build(descs, groups or [0] * n, variants, slots or list(range(n)), flags)
    _, _, ms, ws_bytes = G.goldy_schedule_query(s)
    dA = [a.cuda() for a in As]
    dB = [b.cuda() for b in Bs]
    dC = [torch.full((c_elems[i],), fill, dtype=TORCH_OUT[o], device="cuda") for i, o in enumerate(outs)]
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    streams = [torch.cuda.Stream() for _ in range(max(1, ms))]
    streams[0].wait_stream(torch.cuda.current_stream())
    G.goldy_run(s, [a.data_ptr() for a in dA], [b.data_ptr() for b in dB], [c.data_ptr() for c in dC],
                ws.data_ptr(), ws_bytes, [x.cuda_stream for x in streams])
    torch.cuda.current_stream().wait_stream(streams[0])
    torch.cuda.synchronize()
    assert G.goldy_device_error(clear=True) == 0
    return [c.cpu() for c in dC]


def packed(batch, M, N, K, out, seed):
    a, b = batched_inputs(batch, M, N, K, seed)
    d = G.desc(M, N, K, out, batch=batch)
    return d, a, b, batch * M * N


def check_entries(c_flat, a, b, M, N, stride_c, label):
    for i in range(a.shape[0]):
        got = c_flat[i * stride_c: i * stride_c + M * N].view(M, N)
        check_close(got, a[i], b[i], f"{label} entry {i}")


@pytest.mark.parametrize("kind", list(range(11)))
def test_each_kind_batched(cuda_ok, kind):
    M, N, K = (40, 296, 320) if kind in SWAP_KINDS else (200, 320, 448)
    if kind == 10:
        M, N, K = 300, 520, 448
    for out in (F32, BF16):
        d, a, b, ce = packed(3, M, N, K, out, 70 + kind)
        (c,) = run([d], [a], [b], [out], [vid(kind)], c_elems=[ce])
        check_entries(c, a, b, M, N, M * N, f"kind {kind} out {out}")


@pytest.mark.parametrize("kind,split,rc", [(2, 4, 4), (0, 2, 1), (1, 8, 2), (6, 2, 1), (3, 4, 1)])
def test_batched_split_k(cuda_ok, kind, split, rc):
    M, N, K = (48, 384, 1536) if kind in SWAP_KINDS else (128, 512, 2048)
    d, a, b, ce = packed(5, M, N, K, BF16, 500 + kind)
    (c,) = run([d], [a], [b], [BF16], [vid(kind, split, rc)], c_elems=[ce])
    check_entries(c, a, b, M, N, M * N, f"split {split} kind {kind}")


def test_fused_launch_mixes_batched_and_plain(cuda_ok):
    # one fused launch (same kind): a batch of 4, a plain GEMM, a batch of 2
    shapes = [(4, 128, 256, 512), (1, 200, 256, 320), (2, 64, 256, 1024)]
    descs, As, Bs, ce = [], [], [], []
    for j, (bt, M, N, K) in enumerate(shapes):
        d, a, b, n = packed(bt, M, N, K, F32, 900 + 10 * j)
        descs.append(d)
        As.append(a)
        Bs.append(b)
        ce.append(n)
    for v in (vid(2, 1, 1), vid(2, 4, 1), vid(3, 2, 2)):
        got = run(descs, As, Bs, [F32] * 3, [v] * 3, slots=[0, 1, 2], flags=G.GOLDY_PLAN_FUSED, c_elems=ce)
        for j, (bt, M, N, K) in enumerate(shapes):
            check_entries(got[j], As[j], Bs[j], M, N, M * N, f"fused variant {v} gemm {j}")


@pytest.mark.parametrize("kind", [2, 6, 10])
def test_gapped_strides_leave_gaps_untouched(cuda_ok, kind):
    batch, M, N, K = 3, 130, 264, 192
    if kind in SWAP_KINDS:
        M = 40
    lda, ldb, ldc = K + 8, N + 8, N + 4
    sa, sb, sc = M * lda + 64, K * ldb + 128, M * ldc + 36
    a, b = batched_inputs(batch, M, N, K, 1234 + kind)
    A = torch.zeros(batch * sa, dtype=torch.bfloat16)
    B = torch.zeros(batch * sb, dtype=torch.bfloat16)
    for i in range(batch):
        A[i * sa: i * sa + M * lda].view(M, lda)[:, :K] = a[i]
        B[i * sb: i * sb + K * ldb].view(K, ldb)[:, :N] = b[i]
    d = G.desc(M, N, K, F32, lda=lda, ldb=ldb, ldc=ldc, batch=batch, stride_a=sa, stride_b=sb, stride_c=sc)
    (c,) = run([d], [A], [B], [F32], [vid(kind)], c_elems=[batch * sc], fill=-7.0)
    written = torch.zeros(batch * sc, dtype=torch.bool)
    for i in range(batch):
        blk = c[i * sc: i * sc + M * ldc].view(M, ldc)
        check_close(blk[:, :N].contiguous(), a[i], b[i], f"gapped kind {kind} entry {i}")
        written[i * sc: i * sc + M * ldc].view(M, ldc)[:, :N] = True
    assert torch.all(c[~written] == -7.0)


def test_batched_k_zero(cuda_ok):
    for sc_pad in (0, 20):
        M, N = 33, 70
        ldc = N
        sc = M * ldc + sc_pad
        d = G.desc(M, N, 0, F32, lda=8, ldb=N + 2, ldc=ldc, batch=4, stride_a=M * 8, stride_b=0, stride_c=sc)
        (c,) = run([d], [torch.zeros(8, dtype=torch.bfloat16)], [torch.zeros(8, dtype=torch.bfloat16)], [F32],
                   [vid(2)], c_elems=[4 * sc], fill=5.0)
        for i in range(4):
            assert torch.all(c[i * sc: i * sc + M * N] == 0.0)
            assert torch.all(c[i * sc + M * N: (i + 1) * sc] == 5.0)


@pytest.mark.parametrize("members,i", [(2, 0), (2, 1), (4, 1), (4, 3)])
def test_batched_study_sets_through_the_planner(cuda_ok, members, i):
    st = wl.make_batched_set(i, members)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype, batch=s.batch) for s in st.specs]
    sched = G.goldy_plan(descs, G.goldy_lut_load(), G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
    dA = [a.cuda() for a in st.a]
    dB = [b.cuda() for b in st.b]
    dC = [torch.full((s.batch, s.M, s.N), float("nan"), dtype=torch.bfloat16, device="cuda") for s in st.specs]
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    streams = [torch.cuda.Stream() for _ in range(max(1, ms))]
    streams[0].wait_stream(torch.cuda.current_stream())
    G.goldy_run(sched, [a.data_ptr() for a in dA], [b.data_ptr() for b in dB], [c.data_ptr() for c in dC],
                ws.data_ptr(), ws_bytes, [x.cuda_stream for x in streams])
    torch.cuda.current_stream().wait_stream(streams[0])
    torch.cuda.synchronize()
    assert G.goldy_device_error(clear=True) == 0
    rng = np.random.default_rng(i)
    for j, s in enumerate(st.specs):
        c = dC[j].cpu()
        for e in sorted(set(rng.integers(0, s.batch, size=3).tolist()) | {0, s.batch - 1}):
            rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=4)]))
            check_rows(c[e], st.a[j][e], st.b[j][e], rows, f"study {members}x{i} gemm {j} entry {e}")

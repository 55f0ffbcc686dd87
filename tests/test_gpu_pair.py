"""GPU parity of the CTA-pair GO-Kernel (256 x 256 tiles, one tcgen05 MMA
across two SMs): ragged shapes against the fp64 oracle, exact integer
results, K splits reduced through the workspace, several GEMMs in one fused
launch, and bit-identical results alone vs co-scheduled."""
import numpy as np
import pytest
import torch

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import Launch, check_close, check_rows, run_explicit

pytestmark = pytest.mark.gpu

F32, BF16 = G.GOLDY_F32, G.GOLDY_BF16
PAIR = 10


def vid(split=1, rc=1):
    return G.variant_id(PAIR, split, rc)


def inputs(M, N, K, seed, dist="uniform", scale=1.0):
    return (wl.random_matrix(M, K, seed, dist, scale), wl.random_matrix(K, N, seed + 1, dist, scale))


def test_pair_first_light(cuda_ok):
    a, b = inputs(256, 256, 512, seed=1000)
    (c,) = run_explicit([a], [b], [F32], [vid()])
    check_close(c, a, b, "pair 256x256x512")


@pytest.mark.parametrize("out", [F32, BF16])
@pytest.mark.parametrize("M,N,K", [(300, 320, 448), (512, 768, 1024), (130, 256, 200), (1000, 520, 64)])
def test_pair_ragged(cuda_ok, M, N, K, out):
    a, b = inputs(M, N, K, seed=M + N + K)
    (c,) = run_explicit([a], [b], [out], [vid()])
    check_close(c, a, b, f"pair {M}x{N}x{K}")


def test_pair_integer_exact(cuda_ok):
    a = wl.integer_matrix(384, 512, seed=31)
    b = wl.integer_matrix(512, 640, seed=32)
    (c,) = run_explicit([a], [b], [F32], [vid()])
    exact = (a.to(torch.int64) @ b.to(torch.int64)).to(torch.float32)
    assert torch.equal(c, exact)


def test_pair_grid_cap_is_bit_exact(cuda_ok):
    a, b = inputs(1024, 1024, 512, seed=40)
    outs = [run_explicit([a], [b], [F32], [vid(1, rc)])[0] for rc in (1, 2, 4)]
    check_close(outs[0], a, b, "pair rc1")
    for o in outs[1:]:
        assert torch.equal(outs[0], o)


@pytest.mark.parametrize("out", [F32, BF16])
@pytest.mark.parametrize("split", [2, 4, 8])
@pytest.mark.parametrize("M,N,K", [(300, 320, 1472), (1024, 768, 2048), (130, 520, 448)])
def test_pair_split_k(cuda_ok, M, N, K, split, out):
    # split-K for the pair kind: every CTA publishes its partial, the last
    # split to arrive sums them in split order; ragged tails, splits clamped
    # to the K blocks (448 = 7 blocks), grid caps bit-exact, the workspace's
    # counters back at zero after each run (a second run gives the same bytes)
    a, b = inputs(M, N, K, seed=M + 3 * N + K + split, dist="normal", scale=0.5)
    d = G.desc(M, N, K, out)
    runs = []
    for rc in (1, 4):
        s = G.goldy_schedule_build([d], [0], [vid(split, rc)], [0])
        L = Launch(s, [a], [b], [out])
        for _ in range(2):
            L.run()
            runs.append(L.results()[0])
    check_close(runs[0], a, b, f"pair split {split} {M}x{N}x{K}")
    for r in runs[1:]:
        x, y = (r, runs[0]) if r.dtype != torch.bfloat16 else (r.view(torch.int16), runs[0].view(torch.int16))
        assert torch.equal(x, y)


def test_pair_split_k_integer_exact_and_fused_with_others(cuda_ok):
    # small integers are exact whatever the split; a fused launch of the pair
    # kind with GEMMs of different splits (workspace partials of each) gives
    # the bytes each gives alone
    a = wl.integer_matrix(384, 2048, seed=33)
    b = wl.integer_matrix(2048, 512, seed=34)
    (c,) = run_explicit([a], [b], [F32], [vid(4, 1)])
    assert torch.equal(c, (a.to(torch.int64) @ b.to(torch.int64)).to(torch.float32))
    shapes = [(512, 1024, 2048), (300, 512, 1024), (256, 256, 512)]
    A, B = zip(*[inputs(M, N, K, seed=60 + i, dist="normal", scale=0.1) for i, (M, N, K) in enumerate(shapes)])
    vs = [vid(2, 1), vid(4, 1), vid(1, 1)]
    alone = [run_explicit([A[i]], [B[i]], [F32], [vs[i]])[0] for i in range(3)]
    descs = [G.desc(M, N, K, F32) for (M, N, K) in shapes]
    s = G.goldy_schedule_build(descs, [0, 0, 0], vs, [0, 1, 2], G.GOLDY_PLAN_FUSED)
    L = Launch(s, list(A), list(B), [F32] * 3)
    for _ in range(2):
        L.run()
        got = L.results()
        for i in range(3):
            check_close(got[i], A[i], B[i], f"fused pair {i}")
            assert torch.equal(got[i], alone[i])


def test_pair_fused_and_co_scheduled(cuda_ok):
    shapes = [(512, 1024, 1024), (256, 512, 2048), (768, 256, 512)]
    A, B = zip(*[inputs(M, N, K, seed=50 + i, dist="normal", scale=0.1) for i, (M, N, K) in enumerate(shapes)])
    outs = [F32, BF16, F32]
    vs = [vid(1, 2), vid(1, 4), vid(1, 1)]
    alone = [run_explicit([A[i]], [B[i]], [outs[i]], [vs[i]])[0] for i in range(3)]
    descs = [G.desc(M, N, K, o) for (M, N, K), o in zip(shapes, outs)]
    for flags in (0, G.GOLDY_PLAN_FUSED):
        s = G.goldy_schedule_build(descs, [0, 0, 0], vs, [0, 1, 2], flags)
        L = Launch(s, list(A), list(B), outs)
        L.run()
        got = L.results()
        for i in range(3):
            check_close(got[i], A[i], B[i], f"pair set {i} flags {flags}")
            x, y = got[i], alone[i]
            if x.dtype == torch.bfloat16:
                x, y = x.view(torch.int16), y.view(torch.int16)
            assert torch.equal(x, y)


def test_pair_big_gemm_sampled(cuda_ok):
    st = wl.make_config("hetero_pair")
    (c,) = run_explicit([st.a[3]], [st.b[3]], [F32], [vid()])
    rng = np.random.default_rng(7)
    rows = np.sort(rng.choice(2048, size=40, replace=False))
    rows[0], rows[-1] = 0, 2047
    check_rows(c, st.a[3], st.b[3], rows, "pair 2048x8192x2048")

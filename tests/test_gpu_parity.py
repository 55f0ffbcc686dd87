"""GPU parity: every GO-Kernel variant family against the fp64 oracle, through
the C ABI, on seeded inputs that span several tiles and ragged tails; exact
results on integer inputs; bit-identical results alone vs co-scheduled."""
import numpy as np
import pytest
import torch

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import Launch, check_close, check_rows, run_explicit

pytestmark = pytest.mark.gpu

F32, BF16 = G.GOLDY_F32, G.GOLDY_BF16
KINDS = list(range(10))
SWAP_KINDS = {6, 7, 8, 9}


def vid(kind, split=1, rc=1):
    return G.variant_id(kind, split, rc)


def inputs(M, N, K, seed, dist="uniform", scale=1.0):
    return (wl.random_matrix(M, K, seed, dist, scale), wl.random_matrix(K, N, seed + 1, dist, scale))


def test_first_light_single_gemm(cuda_ok):
    a, b = inputs(256, 256, 512, seed=0)
    (c,) = run_explicit([a], [b], [F32], [vid(2)])
    check_close(c, a, b, "n128_full 256x256x512")


@pytest.mark.parametrize("out", [F32, BF16])
@pytest.mark.parametrize("kind", KINDS)
def test_each_kind_ragged(cuda_ok, kind, out):
    # non-swap: M = 128 + 72 rows, N = 320 (ragged against 64/128/256 tiles), K = 7 blocks
    # swap:     M = 40 (ragged against 32/64-row tiles), N = 296 = 2 x 128 + 40
    M, N, K = (40, 296, 320) if kind in SWAP_KINDS else (200, 320, 448)
    a, b = inputs(M, N, K, seed=10 + kind)
    (c,) = run_explicit([a], [b], [out], [vid(kind)])
    check_close(c, a, b, f"kind {kind} out {out}")


@pytest.mark.parametrize("split", [2, 4, 8])
@pytest.mark.parametrize("kind", [0, 2, 3, 5, 6, 8, 9])
def test_split_k(cuda_ok, kind, split):
    M, N, K = (48, 256, 1024) if kind in SWAP_KINDS else (130, 256, 1024)
    a, b = inputs(M, N, K, seed=100 + kind * 10 + split)
    (c,) = run_explicit([a], [b], [F32], [vid(kind, split)])
    check_close(c, a, b, f"kind {kind} split {split}")
    (c1,) = run_explicit([a], [b], [F32], [vid(kind, 1)])
    # different split -> different summation order; both within the bar
    check_close(c1, a, b, f"kind {kind} split 1")


@pytest.mark.parametrize("kind", [0, 2, 4, 7, 8])
def test_integer_inputs_exact(cuda_ok, kind):
    # |a|,|b| <= 8, K <= 512: every partial sum is an integer < 2^24, exact in fp32
    M, N, K = (64, 384, 512) if kind in SWAP_KINDS else (192, 384, 512)
    a = wl.integer_matrix(M, K, seed=5 + kind)
    b = wl.integer_matrix(K, N, seed=6 + kind)
    for split in (1, 4):
        (c,) = run_explicit([a], [b], [F32], [vid(kind, split)])
        exact = (a.to(torch.int64) @ b.to(torch.int64)).to(torch.float32)
        assert torch.equal(c, exact), f"kind {kind} split {split}"


@pytest.mark.parametrize("kind", [1, 2, 7])
def test_k_tail_and_odd_m(cuda_ok, kind):
    M, N, K = (17, 256, 200) if kind in SWAP_KINDS else (129, 192, 200)
    a, b = inputs(M, N, K, seed=200 + kind)
    (c,) = run_explicit([a], [b], [F32], [vid(kind, 2)])
    check_close(c, a, b, f"kind {kind} K tail")


@pytest.mark.parametrize("kind", [0, 2, 3, 6, 8])
def test_grid_cap_is_bit_exact(cuda_ok, kind):
    # the resource constraint changes how many CTAs share the units, never the math
    M, N, K = (64, 4096, 512) if kind in SWAP_KINDS else (512, 1024, 512)
    a, b = inputs(M, N, K, seed=300 + kind)
    outs = [run_explicit([a], [b], [F32], [vid(kind, 2, rc)])[0] for rc in (1, 2, 4)]
    check_close(outs[0], a, b, "rc 1")
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_co_schedule_invariance(cuda_ok):
    # GEMM 0 alone vs next to three others on four streams vs after them:
    # its bytes must not change (fixed per-element summation order)
    shapes = [(256, 1024, 1024), (128, 1024, 4096), (32, 4096, 1024), (512, 512, 2048)]
    vs = [vid(3, 2, 2), vid(1, 4, 4), vid(7, 2, 4), vid(5, 1, 2)]
    outs = [F32, BF16, F32, F32]
    A, B = zip(*[inputs(M, N, K, seed=400 + i) for i, (M, N, K) in enumerate(shapes)])
    alone = [run_explicit([A[i]], [B[i]], [outs[i]], [vs[i]])[0] for i in range(4)]
    conc = run_explicit(list(A), list(B), outs, vs, groups=[0, 0, 0, 0], slots=[0, 1, 2, 3])
    seq = run_explicit(list(A), list(B), outs, vs, groups=[0, 1, 2, 3], slots=[0, 0, 0, 0])
    mixed = run_explicit(list(A), list(B), outs, vs, groups=[0, 0, 1, 1], slots=[0, 1, 1, 0])
    for i in range(4):
        check_close(alone[i], A[i], B[i], f"gemm {i}")
        for other in (conc, seq, mixed):
            assert torch.equal(alone[i].view(torch.uint8) if alone[i].dtype == torch.bfloat16 else alone[i],
                               other[i].view(torch.uint8) if other[i].dtype == torch.bfloat16 else other[i])


def test_repeat_runs_reuse_workspace(cuda_ok):
    # split-K counters must return to zero: five runs in a row give the same bytes
    a, b = inputs(128, 1024, 4096, seed=500, dist="normal", scale=0.02)
    s = G.goldy_schedule_build([G.desc(128, 1024, 4096, BF16)], [0], [vid(1, 8, 1)], [0])
    L = Launch(s, [a], [b], [BF16])
    L.run()
    first = L.results()[0].clone()
    check_close(first, a, b, "split 8")
    for _ in range(4):
        L.dC[0].fill_(float("nan"))
        L.run()
        assert torch.equal(L.results()[0].view(torch.int16), first.view(torch.int16))


def test_graph_replay_matches_eager(cuda_ok):
    shapes = [(128, 1024, 4096)] * 4
    A, B = zip(*[inputs(M, N, K, seed=600 + i, dist="normal", scale=0.02) for i, (M, N, K) in enumerate(shapes)])
    vs = [vid(1, 4, 4)] * 4
    descs = [G.desc(M, N, K, BF16) for (M, N, K) in shapes]
    s = G.goldy_schedule_build(descs, [0] * 4, vs, [0, 1, 2, 3])
    L = Launch(s, list(A), list(B), [BF16] * 4)
    L.run()
    eager = [c.clone() for c in L.results()]
    g = L.graph()
    for c in L.dC:
        c.fill_(float("nan"))
    for _ in range(3):
        G.goldy_graph_launch(g, L.streams[0].cuda_stream)
    torch.cuda.current_stream().wait_stream(L.streams[0])
    got = L.results()
    for e, x in zip(eager, got):
        assert torch.equal(e.view(torch.int16), x.view(torch.int16))


@pytest.mark.parametrize("fused", [False, True])
def test_exec_replay_matches_eager(cuda_ok, fused):
    """A prepared run (recorded once, replayed with plain launches) gives the
    eager run's bits, over several replays, on split-K, cluster and pair
    variants with a degenerate member in the set."""
    shapes = [(128, 1024, 4096), (256, 512, 2048), (100, 384, 1000), (0, 128, 64)]
    A, B = zip(*[inputs(M, N, K, seed=650 + i, dist="normal", scale=0.02) for i, (M, N, K) in enumerate(shapes)])
    vs = [vid(1, 4, 4), vid(10, 1, 4), vid(3, 2, 4), vid(2)]
    descs = [G.desc(M, N, K, BF16) for (M, N, K) in shapes]
    s = G.goldy_schedule_build(descs, [0] * 4, vs, [0, 1, 2, 3], G.GOLDY_PLAN_FUSED if fused else 0)
    L = Launch(s, list(A), list(B), [BF16] * 4)
    L.run()
    eager = [c.clone() for c in L.results()]
    L.streams[0].wait_stream(torch.cuda.current_stream())
    x = L.exec()
    for c in L.dC:
        c.fill_(float("nan"))
    L.streams[0].wait_stream(torch.cuda.current_stream())
    for _ in range(3):
        G.goldy_exec_launch(x)
    torch.cuda.current_stream().wait_stream(L.streams[0])
    got = L.results()
    for e, g in zip(eager, got):
        assert torch.equal(e.view(torch.int16), g.view(torch.int16))
    check_close(got[1].float(), A[1], B[1], "exec pair")
    del x


def test_degenerate_sizes(cuda_ok):
    a0 = torch.zeros((0, 64), dtype=torch.bfloat16)
    b0 = wl.random_matrix(64, 128, seed=1)
    ak = torch.zeros((70, 0), dtype=torch.bfloat16)
    bk = torch.zeros((0, 136), dtype=torch.bfloat16)
    a, b = inputs(33, 64, 64, seed=3)
    descs = [G.desc(0, 128, 64), G.desc(70, 136, 0, lda=8), G.desc(33, 64, 64)]
    s = G.goldy_schedule_build(descs, [0, 0, 0], [vid(2), vid(2), vid(6)], [0, 1, 2])
    L = Launch(s, [a0, ak, a], [b0, bk, b], [F32, F32, F32])
    L.run()
    c0, ck, c = L.results()
    assert c0.shape == (0, 128)
    assert torch.equal(ck, torch.zeros_like(ck))
    check_close(c, a, b, "small after degenerate")


@pytest.mark.parametrize("name", ["pair_256", "ffn_slices", "lstm_gates"])
def test_config_full_size(cuda_ok, name):
    st = wl.make_config(name)
    n = len(st.specs)
    kinds = {"pair_256": 3, "ffn_slices": 1, "lstm_gates": 7}
    split = {"pair_256": 1, "ffn_slices": 4, "lstm_gates": 2}
    v = vid(kinds[name], split[name], 4)
    outs = [s.out_dtype for s in st.specs]
    got = run_explicit(st.a, st.b, outs, [v] * n, slots=list(range(n)))
    for i in range(n):
        check_close(got[i], st.a[i], st.b[i], f"{name}[{i}]")


def test_config_hetero_pair_sampled(cuda_ok):
    st = wl.make_config("hetero_pair")
    vs = [vid(3, 1, 4)] * 3 + [vid(4, 1, 1)]
    got = run_explicit(st.a, st.b, [F32] * 4, vs, slots=[0, 1, 2, 3])
    for i in range(3):
        check_close(got[i], st.a[i], st.b[i], f"small[{i}]")
    rng = np.random.default_rng(3)
    rows = np.sort(rng.choice(2048, size=48, replace=False))
    rows[0], rows[-1] = 0, 2047
    check_rows(got[3], st.a[3], st.b[3], rows, "big sampled rows")


def test_device_error_word_clear(cuda_ok):
    assert G.goldy_device_error(clear=False) == 0


def _run_sched(As, Bs, outs, variants, groups, slots, flags):
    descs = [G.desc(a.shape[0], b.shape[1], a.shape[1], o) for a, b, o in zip(As, Bs, outs)]
    s = G.goldy_schedule_build(descs, groups, variants, slots, flags)
    L = Launch(s, As, Bs, outs)
    L.run()
    return L.results()


def _same_bytes(x, y):
    if x.dtype == torch.bfloat16:
        return torch.equal(x.view(torch.int16), y.view(torch.int16))
    return torch.equal(x, y)


def test_fused_launch_matches_streams(cuda_ok):
    # four same-kind GEMMs of different shapes and splits in one launch
    shapes = [(128, 1024, 4096), (100, 512, 1024), (256, 320, 2048), (128, 1024, 4096)]
    A, B = zip(*[inputs(M, N, K, seed=700 + i, dist="normal", scale=0.05) for i, (M, N, K) in enumerate(shapes)])
    vs = [vid(1, 4, 4), vid(1, 2, 2), vid(1, 1, 1), vid(1, 8, 4)]
    outs = [BF16] * 4
    ref = _run_sched(list(A), list(B), outs, vs, [0] * 4, [0, 1, 2, 3], 0)
    got = _run_sched(list(A), list(B), outs, vs, [0] * 4, [0, 1, 2, 3], G.GOLDY_PLAN_FUSED)
    for i in range(4):
        check_close(got[i], A[i], B[i], f"fused gemm {i}")
        assert _same_bytes(got[i], ref[i])


def test_fused_mixed_kinds_waves_and_degenerate(cuda_ok):
    # group 0: CD 3 over 5 members -> waves {0,1,2} (three kinds, three launches) and
    # {3,4} (one kind: one fused launch); group 1: a K = 0 member next to a real one
    shapes = [(64, 4096, 512), (200, 320, 448), (40, 296, 320), (200, 320, 448), (130, 256, 1024),
              (70, 136, 0), (33, 64, 64)]
    outs = [F32, F32, BF16, F32, F32, F32, F32]
    A, B = [], []
    for i, (M, N, K) in enumerate(shapes):
        if K == 0:
            A.append(torch.zeros((M, 0), dtype=torch.bfloat16))
            B.append(torch.zeros((0, N), dtype=torch.bfloat16))
        else:
            a, b = inputs(M, N, K, seed=800 + i)
            A.append(a)
            B.append(b)
    vs = [vid(7, 2, 4), vid(3, 1, 2), vid(6, 1, 4), vid(3, 2, 2), vid(3, 4, 4), vid(2), vid(2)]
    groups = [0, 0, 0, 0, 0, 1, 1]
    slots = [0, 1, 2, 0, 1, 0, 1]
    descs = [G.desc(a.shape[0], b.shape[1], a.shape[1], o, lda=max(8, a.shape[1])) for a, b, o in zip(A, B, outs)]
    res = {}
    for flags in (0, G.GOLDY_PLAN_FUSED):
        s = G.goldy_schedule_build(descs, groups, vs, slots, flags)
        L = Launch(s, A, B, outs)
        L.run()
        res[flags] = L.results()
    for i in range(7):
        if shapes[i][2] == 0:
            assert torch.equal(res[G.GOLDY_PLAN_FUSED][i], torch.zeros_like(res[0][i]))
            continue
        check_close(res[G.GOLDY_PLAN_FUSED][i], A[i], B[i], f"fused mixed {i}")
        assert _same_bytes(res[G.GOLDY_PLAN_FUSED][i], res[0][i])


def test_fused_plan_graph_replay(cuda_ok):
    st = wl.make_config("lstm_gates")
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    v = vid(7, 2, 4)
    s = G.goldy_schedule_build(descs, [0] * 8, [v] * 8, list(range(8)), G.GOLDY_PLAN_FUSED)
    L = Launch(s, st.a, st.b, [s_.out_dtype for s_ in st.specs])
    g = L.graph()
    for _ in range(3):
        G.goldy_graph_launch(g, L.streams[0].cuda_stream)
    torch.cuda.current_stream().wait_stream(L.streams[0])
    got = L.results()
    for i in range(8):
        check_close(got[i], st.a[i], st.b[i], f"lstm fused {i}")


def test_phase_trace_is_consistent(cuda_ok):
    # the optional per-CTA trace: every CTA stamps its phases in order and the
    # units it reports add up to the launch's units
    shapes = [(128, 1024, 4096)] * 2
    A, B = zip(*[inputs(M, N, K, seed=900 + i, dist="normal", scale=0.05) for i, (M, N, K) in enumerate(shapes)])
    v = vid(1, 4, 1)
    descs = [G.desc(M, N, K, BF16) for (M, N, K) in shapes]
    s = G.goldy_schedule_build(descs, [0, 0], [v, v], [0, 1], G.GOLDY_PLAN_FUSED)
    L = Launch(s, list(A), list(B), [BF16, BF16])
    trace = torch.zeros(512 * 16, dtype=torch.int64, device="cuda")
    A_, B_, C_ = L.ptrs()
    G.goldy_run_ex(s, A_, B_, C_, L.ws.data_ptr(), L.ws_bytes, [x.cuda_stream for x in L.streams],
                   trace=trace.data_ptr(), trace_ctas=512)
    got = L.results()
    for i in range(2):
        check_close(got[i], A[i], B[i], f"traced {i}")
    t = trace.view(512, 16).cpu()
    rows = t[t[:, 0] != 0]
    assert rows.shape[0] > 0
    assert int(rows[:, 14].sum()) == 2 * 16 * 4                  # 16 tiles x split 4 per GEMM
    for r in rows.tolist():
        # slot 1 is stamped by the first epilogue thread, slots 2-4 by the
        # producer and the MMA thread: ordered within each thread's sequence
        assert r[0] <= r[1] <= r[5] and r[0] <= r[2] <= r[3] <= r[4] <= r[5] <= r[8] <= r[9]
        assert r[6] <= r[7]


@pytest.mark.parametrize("j", [0, 17, 63])
def test_sweep_sets_through_the_planner(cuda_ok, j):
    # randomized sets (2-16 GEMMs, M 16-4096, N, K 256-8192) through the
    # packaged table in fused mode; sampled rows of every GEMM vs the oracle
    st = wl.make_sweep_set(j)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    sched = G.goldy_plan(descs, G.goldy_lut_load(G.DEFAULT_LUT), G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    L = Launch(sched, st.a, st.b, [s.out_dtype for s in st.specs])
    L.run()
    got = L.results()
    rng = np.random.default_rng(j)
    for i, s in enumerate(st.specs):
        rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=min(6, s.M))]))
        check_rows(got[i], st.a[i], st.b[i], rows, f"sweep {j} gemm {i} {s.M}x{s.N}x{s.K}")


@pytest.mark.parametrize("j", [0, 8, 33])
def test_sweep_sets_through_the_predictor_plan(cuda_ok, j):
    # sets whose schedule changes when the trained CD predictor (Eq. 1)
    # supplies the preferences: sampled rows of every GEMM vs the oracle
    st = wl.make_sweep_set(j)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    lut = G.goldy_lut_load(G.DEFAULT_LUT)
    sched = G.goldy_plan_ex(descs, lut, G.goldy_predictor_load(), G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    L = Launch(sched, st.a, st.b, [s.out_dtype for s in st.specs])
    L.run()
    got = L.results()
    rng = np.random.default_rng(100 + j)
    for i, s in enumerate(st.specs):
        rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=min(6, s.M))]))
        check_rows(got[i], st.a[i], st.b[i], rows, f"sweep {j} (predictor plan) gemm {i} {s.M}x{s.N}x{s.K}")


@pytest.mark.parametrize("j", [12, 14, 17])
def test_one_kind_per_wave_plans_match_oracle(cuda_ok, j):
    # randomized sets in which the planner moves GEMMs of a wave to the kind
    # of the wave's largest GEMM (set 12: two into the CTA-pair kernel, 14:
    # seven between single-CTA kinds, 17: four into the pair kernel): every
    # GEMM on sampled rows (first and last included) against the oracle, the
    # plan bit-identical fused, in streams mode and as a prepared run
    st = wl.make_sweep_set(j)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    lut = G.goldy_lut_load(G.DEFAULT_LUT)
    fused = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    classes = (1, 2, 4, 8, 16)
    moved = 0
    for i, d in enumerate(descs):
        _, v, _, cd = G.goldy_schedule_entry(fused, i)
        table_v = G.goldy_lut_lookup(lut, d)[1][next(k for k, c in enumerate(classes) if c >= cd)]
        moved += int(v != table_v)
    assert moved >= 2
    outs = [s.out_dtype for s in st.specs]
    Lf = Launch(fused, st.a, st.b, outs)
    Lf.run()
    got = Lf.results()
    rng = np.random.default_rng(4000 + j)
    for i, s in enumerate(st.specs):
        rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=min(8, s.M))]))
        check_rows(got[i], st.a[i], st.b[i], rows, f"sweep {j} gemm {i} {s.M}x{s.N}x{s.K}")
    streams = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO)
    Ls = Launch(streams, st.a, st.b, outs)
    Ls.run()
    for x, y in zip(got, Ls.results()):
        assert torch.equal(x.view(torch.uint8), y.view(torch.uint8))
    for c in Lf.dC:
        c.fill_(float("nan"))
    x = Lf.exec()
    G.goldy_exec_launch(x)
    for a, b in zip(got, Lf.results()):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
    del x


@pytest.mark.parametrize("j", [30, 48, 16])
def test_few_launch_runs_on_one_stream_match(cuda_ok, j):
    # randomized sets whose fused plan has 2 to 5 launches: with inputs_ready
    # they (like every fused run) go out on streams[0] alone, each wave's
    # largest first; replayed back to back as prepared runs they give the
    # same bytes as the forked multi-stream run without the option, and the
    # oracle's values
    st = wl.make_sweep_set(j)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    sched = G.goldy_plan(descs, G.goldy_lut_load(G.DEFAULT_LUT), G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    outs = [s.out_dtype for s in st.specs]
    L = Launch(sched, st.a, st.b, outs)
    L.run()
    ref = L.results()
    rng = np.random.default_rng(5000 + j)
    for i, s in enumerate(st.specs):
        rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=min(6, s.M))]))
        check_rows(ref[i], st.a[i], st.b[i], rows, f"sweep {j} gemm {i}")
    for c in L.dC:
        c.fill_(float("nan"))
    A, B, C = L.ptrs()
    x = G.goldy_exec_create(sched, A, B, C, L.ws.data_ptr(), L.ws_bytes, [s.cuda_stream for s in L.streams],
                            inputs_ready=True)
    for _ in range(4):
        G.goldy_exec_launch(x)
    got = L.results()
    for a, b in zip(got, ref):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
    del x


@pytest.mark.parametrize("fused", [False, True])
def test_dependent_launches_see_the_previous_kernels_output(cuda_ok, fused):
    """Kernels of one stream overlap their set-up with the previous kernel
    (programmatic dependent launch) but must read its results: a chain of
    GEMMs, each reading the previous one's bf16 output as its A, run one after
    another on one stream, matches the oracle chain, bit-identical to plain
    serialised launches."""
    M, N, K = 256, 512, 512
    a0 = wl.random_matrix(M, K, 77, "normal", 0.05)
    bs = [wl.random_matrix(K, N, 78 + j, "normal", 0.05) for j in range(4)]
    descs = [G.desc(M, N, K, BF16)] * 4
    vs = [vid(2, 1, 1), vid(3, 2, 2), vid(10, 1, 1), vid(2, 4, 4)]
    s = G.goldy_schedule_build(descs, [0, 1, 2, 3], vs, [0, 0, 0, 0], G.GOLDY_PLAN_FUSED if fused else 0)
    _, _, ms, ws_bytes = G.goldy_schedule_query(s)
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    dA0 = a0.cuda()
    dB = [b.cuda() for b in bs]
    outs = {}
    for serial in (False, True):
        dC = [torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(4)]
        A = [dA0.data_ptr()] + [c.data_ptr() for c in dC[:3]]     # GEMM j reads GEMM j-1's output
        st = torch.cuda.Stream()
        st.wait_stream(torch.cuda.current_stream())
        for _ in range(3):
            G.goldy_run_ex(s, A, [b.data_ptr() for b in dB], [c.data_ptr() for c in dC], ws.data_ptr(), ws_bytes,
                           [st.cuda_stream], serial_launch=serial)
        torch.cuda.current_stream().wait_stream(st)
        torch.cuda.synchronize()
        assert G.goldy_device_error(clear=True) == 0
        outs[serial] = [c.cpu() for c in dC]
    prev = a0
    for j in range(4):
        check_close(outs[False][j], prev, bs[j], f"chain step {j}")
        prev = outs[False][j]
        assert torch.equal(outs[False][j].view(torch.int16), outs[True][j].view(torch.int16))


@pytest.mark.parametrize("fused", [False, True])
def test_inputs_ready_runs_overlap_and_match(cuda_ok, fused):
    """With inputs_ready the load and MMA roles of a launch start while the
    previous kernel on the stream is still running; the epilogue still waits
    for it.  Independent GEMMs (none reads another's output) replayed back to
    back on one stream give the same bytes as plain serialised launches and
    the oracle's results."""
    M, N, K = 256, 512, 512
    As = [wl.random_matrix(M, K, 177 + j, "normal", 0.05) for j in range(4)]
    bs = [wl.random_matrix(K, N, 178 + j, "normal", 0.05) for j in range(4)]
    descs = [G.desc(M, N, K, BF16)] * 4
    vs = [vid(2, 1, 1), vid(3, 2, 2), vid(10, 1, 1), vid(2, 4, 4)]
    s = G.goldy_schedule_build(descs, [0, 1, 2, 3], vs, [0, 0, 0, 0], G.GOLDY_PLAN_FUSED if fused else 0)
    _, _, ms, ws_bytes = G.goldy_schedule_query(s)
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    dA = [a.cuda() for a in As]
    dB = [b.cuda() for b in bs]
    outs = {}
    for early in (True, False):
        dC = [torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(4)]
        st = torch.cuda.Stream()
        st.wait_stream(torch.cuda.current_stream())
        for _ in range(5):
            G.goldy_run_ex(s, [a.data_ptr() for a in dA], [b.data_ptr() for b in dB], [c.data_ptr() for c in dC],
                           ws.data_ptr(), ws_bytes, [st.cuda_stream], serial_launch=not early, inputs_ready=early)
        torch.cuda.current_stream().wait_stream(st)
        torch.cuda.synchronize()
        assert G.goldy_device_error(clear=True) == 0
        outs[early] = [c.cpu() for c in dC]
    for j in range(4):
        check_close(outs[True][j], As[j], bs[j], f"independent gemm {j} with inputs_ready")
        assert torch.equal(outs[True][j].view(torch.int16), outs[False][j].view(torch.int16))


def _multi_group_sweep_sets(lut, count):
    """The first `count` randomized sets whose plan has several groups."""
    found = []
    for j in range(wl.SWEEP_SETS):
        _, specs, _ = wl.sweep_specs(j)
        descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in specs]
        if G.goldy_schedule_query(G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED))[1] > 1:
            found.append(j)
            if len(found) == count:
                break
    return found


@pytest.mark.parametrize("pick", [0, 1])
def test_fused_dispatch_matches_strict_groups(cuda_ok, pick):
    # A multi-group plan in fused mode (one fork and join, groups ordered by
    # launch priority, the first wave's largest launch first) against the
    # same plan in streams mode (groups one after another): same bytes, run
    # eagerly, as a prepared run and as a CUDA graph.
    lut = G.goldy_lut_load(G.DEFAULT_LUT)
    picks = _multi_group_sweep_sets(lut, 2)
    assert len(picks) == 2, "want randomized sets whose plan has several groups"
    j = picks[pick]
    st = wl.make_sweep_set(j)
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    fused = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    strict = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO)
    outs = [s.out_dtype for s in st.specs]
    Ls = Launch(strict, st.a, st.b, outs)
    Ls.run()
    ref = Ls.results()
    Lf = Launch(fused, st.a, st.b, outs)
    Lf.run()
    runs = [Lf.results()]
    for make in (Lf.exec, Lf.graph):
        for c in Lf.dC:
            c.fill_(float("nan"))
        handle = make()
        if make == Lf.exec:
            G.goldy_exec_launch(handle)
        else:
            G.goldy_graph_launch(handle, Lf.streams[0].cuda_stream)
        torch.cuda.current_stream().wait_stream(Lf.streams[0])
        runs.append(Lf.results())
        del handle
    for got in runs:
        for i in range(len(descs)):
            x, y = got[i], ref[i]
            if x.dtype == torch.bfloat16:
                x, y = x.view(torch.int16), y.view(torch.int16)
            assert torch.equal(x, y), f"sweep {j} gemm {i}"


def test_phase_trace_regions_per_launch(cuda_ok):
    # A run of several launches traces into consecutive regions, one per
    # launch in launch order: each region's CTAs record its grid size and
    # their index, every CTA stamps its phases in order, and the units over
    # all regions add up to the plan's units.
    lut = G.goldy_lut_load(G.DEFAULT_LUT)
    st = wl.make_sweep_set(_multi_group_sweep_sets(lut, 1)[0])
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    sched = G.goldy_plan(descs, lut, G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)
    L = Launch(sched, st.a, st.b, [s.out_dtype for s in st.specs])
    ctas = 8192
    trace = torch.zeros(ctas * 16, dtype=torch.int64, device="cuda")
    A_, B_, C_ = L.ptrs()
    G.goldy_run_ex(sched, A_, B_, C_, L.ws.data_ptr(), L.ws_bytes, [x.cuda_stream for x in L.streams],
                   trace=trace.data_ptr(), trace_ctas=ctas)
    L.results()
    t = trace.view(ctas, 16).cpu()
    off, regions, units = 0, 0, 0
    while off < ctas and int(t[off, 12]) > 0:
        grid = int(t[off, 12])
        rows = t[off:off + grid]
        assert (rows[:, 12] == grid).all() and (rows[:, 13] == torch.arange(grid)).all()
        for r in rows.tolist():
            # every stamp a CTA wrote lies between its set-up and its exit (the
            # odd CTA of a pair issues no MMAs and leaves those stamps at 0)
            assert 0 < r[0] <= r[1] <= r[9]
            for k in (2, 3, 4, 5, 8):
                assert r[k] == 0 or r[1] <= r[k] <= r[9], (k, r)
            assert r[5] <= r[8]
        units += int(rows[:, 14].sum())
        off += grid
        regions += 1
    assert regions >= 2
    assert int(t[off:, 0].abs().sum()) == 0                     # nothing written past the last region
    expect = 0
    for i in range(len(descs)):
        _, v, _, _ = G.goldy_schedule_entry(sched, i)
        info = G.goldy_variant_info_get(v)
        s = st.specs[i]
        rows_ = info["mma_n"] if info["swap_ab"] else (256 if info["cta_pair"] == 2 else 128)
        cols = 128 if info["swap_ab"] else info["mma_n"]
        tiles = -(-s.M // rows_) * -(-s.N // cols)
        split = min(info["split_k"], -(-s.K // 64))
        expect += tiles * split * (2 if info["cta_pair"] == 2 else 1)   # a pair unit counts on both CTAs
    assert units == expect


def test_fused_launch_with_unequal_units_hands_them_out_dynamically(cuda_ok):
    # One fused launch (kind n64_full, split 1, GPU/4 caps: 76 CTAs) over
    # 64 units of 4 K blocks and 16 units of 32 K blocks: more units than
    # CTAs and lengths 8x apart, so the units are handed out by the launch's
    # counter, longest first.  Results match the oracle and, bit for bit, each
    # GEMM run alone; repeated runs and replays give the same bytes (the last
    # CTA leaves the counter zeroed: a stale counter would skip units and
    # leave the NaN fill in C).
    shapes = [(512, 1024, 256), (256, 512, 2048)]
    A, B = zip(*[inputs(M, N, K, seed=1100 + i) for i, (M, N, K) in enumerate(shapes)])
    v = vid(0, 1, 4)
    alone = [run_explicit([A[i]], [B[i]], [F32], [v])[0] for i in range(2)]
    descs = [G.desc(M, N, K, F32) for (M, N, K) in shapes]
    s = G.goldy_schedule_build(descs, [0, 0], [v, v], [0, 1], G.GOLDY_PLAN_FUSED)
    L = Launch(s, list(A), list(B), [F32, F32])
    for rep in range(3):
        for c in L.dC:
            c.fill_(float("nan"))
        L.run()
        got = L.results()
        for i in range(2):
            if rep == 0:
                check_close(got[i], A[i], B[i], f"dynamic units gemm {i}")
            assert torch.equal(got[i], alone[i]), f"run {rep} gemm {i}"
    ex = L.exec()
    for rep in range(3):
        for c in L.dC:
            c.fill_(float("nan"))
        torch.cuda.synchronize()
        G.goldy_exec_launch(ex)
        got = L.results()
        for i in range(2):
            assert torch.equal(got[i], alone[i]), f"replay {rep} gemm {i}"
    del ex

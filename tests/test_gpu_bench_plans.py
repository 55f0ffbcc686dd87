"""The exact plans the benchmark times, at full size, against the fp64 oracle.

Each fixed set is planned by the dynamic logic (GOLDY_PLAN_AUTO with fused
waves) and run the way bench.py runs it: one prepared run per rotating copy
of the inputs (inputs past twice the L2), replayed back to back with every
launch's set-up overlapping the previous kernel.  After the replays, every
copy's outputs are compared with the oracle: pair_256, ffn_slices and
lstm_gates element by element in full; hetero_pair's three 512 x 1024 x 1024
GEMMs in full and its 2048 x 8192 x 2048 GEMM on 256 seeded rows including
rows 0 and 2047.  Every copy holds the same inputs, so every copy's outputs
must also be byte-identical to copy 0's.  The plans are asserted to be the
ones the bench line reports."""
import numpy as np
import pytest
import torch

import bench
from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import check_close, check_rows

pytestmark = pytest.mark.gpu

# variant names the planner picks for each fixed set (the bench line's plan)
EXPECTED_PLAN = {
    "pair_256": {"n64_full_s4_rc1"},
    "ffn_slices": {"n128_full_s4_rc4"},
    "lstm_gates": {"n128_full_s1_rc2"},
    "hetero_pair": {"p256_pair_s1_rc4"},
}


def _bench_runner(name):
    st = wl.make_config(name)
    lut = G.goldy_lut_load(G.DEFAULT_LUT)
    descs, sched, plan, single = bench.plan_set(G, st, lut, G.GOLDY_PLAN_FUSED)
    names = {G.goldy_variant_info_get(v)["name"] for _, v, _, _ in plan}
    assert names == EXPECTED_PLAN[name], names
    assert single, "every fixed set runs as one fused launch per step"
    l2 = int(getattr(torch.cuda.get_device_properties(0), "L2_cache_size", 126 << 20))
    copies, _ = bench.rotating_copies(st, l2)
    r = bench.SetRunner(st, sched, copies)
    for A, B, C in r.copies:             # outputs start as NaN: unwritten elements fail the check
        for c in C:
            c.fill_(float("nan"))
    torch.cuda.synchronize()
    r.timed(3 * copies)                  # back to back, rotating, as the timed region
    torch.cuda.synchronize()
    assert G.goldy_device_error(clear=True) == 0
    return st, r


@pytest.mark.parametrize("name", ["pair_256", "ffn_slices", "lstm_gates"])
def test_bench_plan_full_size_every_element(cuda_ok, name):
    st, r = _bench_runner(name)
    first = [c.cpu() for c in r.copies[0][2]]
    for i in range(len(st.specs)):
        check_close(first[i], st.a[i], st.b[i], f"{name}[{i}] as benchmarked")
    for k, (_, _, C) in enumerate(r.copies[1:], start=1):
        for i, c in enumerate(C):
            assert torch.equal(c.cpu().view(torch.uint8), first[i].view(torch.uint8)), f"copy {k} gemm {i}"
    del r


def test_bench_plan_hetero_pair(cuda_ok):
    st, r = _bench_runner("hetero_pair")
    first = [c.cpu() for c in r.copies[0][2]]
    big = [i for i, s in enumerate(st.specs) if s.M == 2048]
    assert len(big) == 1
    for i, s in enumerate(st.specs):
        if i in big:
            rng = np.random.default_rng(2409)
            rows = np.sort(rng.choice(np.arange(1, s.M - 1), size=254, replace=False))
            rows = np.concatenate([[0], rows, [s.M - 1]])
            assert len(rows) == 256
            check_rows(first[i], st.a[i], st.b[i], rows, "hetero_pair 2048x8192x2048 as benchmarked")
        else:
            check_close(first[i], st.a[i], st.b[i], f"hetero_pair[{i}] as benchmarked")
    for k, (_, _, C) in enumerate(r.copies[1:], start=1):
        for i, c in enumerate(C):
            assert torch.equal(c.cpu().view(torch.uint8), first[i].view(torch.uint8)), f"copy {k} gemm {i}"
    del r

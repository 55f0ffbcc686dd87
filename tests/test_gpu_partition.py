"""SM partitions (green contexts): the paper's CU-partition study (Sec. 6.9, GOLDYLOC with Resource Partitioning)
runs the whole method inside a quarter, half or all of the GPU.  Schedules
run on a partition's streams give the oracle's results, stay on the
partition's SMs (the per-CTA trace records the SM of every CTA), and a
quarter of the GPU is measurably slower than the whole on tensor-bound work."""
import numpy as np
import pytest
import torch

from paper_2409_02227_gb300 import goldy as G
from paper_2409_02227_gb300 import workloads as wl
from tests.gpu_util import check_rows

pytestmark = pytest.mark.gpu


class PartRun:
    """Device buffers of one set and a prepared run on a partition's streams."""

    def __init__(self, st, sched, part, trace=None, trace_ctas=0):
        _, _, ms, ws_bytes = G.goldy_schedule_query(sched)
        self.ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
        self.A = [a.cuda() for a in st.a]
        self.B = [b.cuda() for b in st.b]
        cdt = [torch.bfloat16 if s.out_dtype == 0 else torch.float32 for s in st.specs]
        self.C = [torch.full((s.M, s.N), float("nan"), dtype=d, device="cuda") for s, d in zip(st.specs, cdt)]
        torch.cuda.synchronize()
        _, streams = G.goldy_partition_query(part, max(1, ms))
        self.x = G.goldy_exec_create(sched, [a.data_ptr() for a in self.A], [b.data_ptr() for b in self.B],
                                     [c.data_ptr() for c in self.C], self.ws.data_ptr(), ws_bytes, streams,
                                     trace=trace or 0, trace_ctas=trace_ctas)

    def time_ms(self, warmup, reps):
        return G.goldy_exec_time([self.x], warmup, reps)


def _plan(st):
    descs = [G.desc(s.M, s.N, s.K, s.out_dtype) for s in st.specs]
    return G.goldy_plan(descs, G.goldy_lut_load(), G.GOLDY_PLAN_AUTO | G.GOLDY_PLAN_FUSED)


@pytest.mark.parametrize("sms", [38, 76, 0])
def test_partition_results_match_oracle(cuda_ok, sms):
    dev_sms = torch.cuda.get_device_properties(0).multi_processor_count
    part = G.goldy_partition_create(sms, 16)
    got_sms, _ = G.goldy_partition_query(part)
    if sms == 0:
        assert got_sms == dev_sms
    else:
        assert sms <= got_sms < dev_sms
    for name in ("ffn_slices", "hetero_pair"):
        st = wl.make_config(name)
        r = PartRun(st, _plan(st), part)
        r.time_ms(0, 1)                               # one replay; synchronises on its end event
        assert G.goldy_device_error(clear=True) == 0
        rng = np.random.default_rng(sms)
        for i, s in enumerate(st.specs):
            rows = np.unique(np.concatenate([[0, s.M - 1], rng.integers(0, s.M, size=4)]))
            check_rows(r.C[i].cpu(), st.a[i], st.b[i], rows, f"{name} gemm {i} in {got_sms}-SM partition")
        del r
    del part


def test_partition_confines_ctas_to_its_sms(cuda_ok):
    part = G.goldy_partition_create(38, 4)
    got_sms, _ = G.goldy_partition_query(part)
    st = wl.make_config("ffn_slices")
    trace = torch.zeros(4096 * 16, dtype=torch.int64, device="cuda")
    r = PartRun(st, _plan(st), part, trace=trace.data_ptr(), trace_ctas=4096)
    r.time_ms(0, 1)
    t = trace.view(4096, 16).cpu()
    rows = t[t[:, 0] != 0]
    assert rows.shape[0] > 0
    sm_ids = set(int(x) for x in rows[:, 15].tolist())
    assert len(sm_ids) <= got_sms, (len(sm_ids), got_sms)
    # every unit of the set was processed inside the partition
    del r, part


def test_quarter_partition_is_slower_on_tensor_bound_work(cuda_ok):
    st = wl.make_config("hetero_pair")
    sched = _plan(st)
    times = {}
    for sms in (38, 0):
        part = G.goldy_partition_create(sms, 16)
        r = PartRun(st, sched, part)
        times[sms] = r.time_ms(5, 20)
        del r, part
    assert G.goldy_device_error(clear=True) == 0
    assert times[38] > 2.0 * times[0], times

"""ctypes binding of ``include/goldy.h`` — argument marshalling only.

Every function here has the name of the C entry point it calls and does no
work of its own beyond converting arguments and raising ``GoldyError`` on a
non-zero status.  Device pointers and CUDA streams are plain integers
(``tensor.data_ptr()``, ``torch.cuda.Stream().cuda_stream``).  The library is
``libgoldy.so`` next to this file, built by ``paper_2409_02227_gb300.build``;
importing this module without it raises ImportError — there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence, Tuple

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgoldy.so")
DEFAULT_LUT = os.path.join(_HERE, "data", "goldy_lut.bin")
DEFAULT_PREDICTOR = os.path.join(_HERE, "data", "goldy_lr.bin")
LR_FEATURES = 18

GOLDY_OK = 0
GOLDY_ERR_INVALID_ARG = 1
GOLDY_ERR_UNSUPPORTED = 2
GOLDY_ERR_LUT = 3
GOLDY_ERR_CUDA = 4
GOLDY_ERR_TIMEOUT = 5
GOLDY_ERR_NOMEM = 6

GOLDY_BF16 = 0
GOLDY_F32 = 1

GOLDY_PLAN_AUTO = 0
GOLDY_PLAN_SEQUENTIAL = 1
GOLDY_PLAN_DEFAULT = 2
GOLDY_PLAN_GO = 3
GOLDY_PLAN_FORCE_CD = 4
GOLDY_PLAN_FUSED = 0x10
GOLDY_MAX_GEMMS = 64
GOLDY_MAX_STREAMS = 16


def force_cd(cd: int) -> int:
    """Flags for GOLDY_PLAN_FORCE_CD with concurrency degree ``cd``."""
    return GOLDY_PLAN_FORCE_CD | (int(cd) << 8)


class GoldyError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        super().__init__(f"{where}: status {status}: {message}")
        self.status = status


class goldy_ewise_desc(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class goldy_gemm_desc(ctypes.Structure):
    _fields_ = [("M", ctypes.c_int64), ("N", ctypes.c_int64), ("K", ctypes.c_int64),
                ("lda", ctypes.c_int64), ("ldb", ctypes.c_int64), ("ldc", ctypes.c_int64),
                ("trans_a", ctypes.c_int32), ("trans_b", ctypes.c_int32),
                ("a_dtype", ctypes.c_int32), ("b_dtype", ctypes.c_int32),
                ("c_dtype", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("batch", ctypes.c_int64), ("stride_a", ctypes.c_int64), ("stride_b", ctypes.c_int64),
                ("stride_c", ctypes.c_int64)]


class goldy_run_opts(ctypes.Structure):
    _fields_ = [("ev_begin", ctypes.POINTER(ctypes.c_void_p)), ("ev_end", ctypes.POINTER(ctypes.c_void_p)),
                ("trace", ctypes.c_void_p), ("trace_ctas", ctypes.c_size_t), ("serial_launch", ctypes.c_int32),
                ("inputs_ready", ctypes.c_int32), ("wait_limit_us", ctypes.c_uint32),
                ("test_stall_first_stage", ctypes.c_int32)]


class goldy_variant_info(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("id", "kind", "mma_m", "mma_n", "swap_ab", "stages", "acc_stages", "tmem_cols",
                 "smem_bytes", "split_k", "rc_div", "ctas_per_sm", "cta_pair")] + [("name", ctypes.c_char * 32)]

    def as_dict(self) -> dict:
        d = {n: getattr(self, n) for n, _ in self._fields_ if n != "name"}
        d["name"] = self.name.decode()
        return d


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'` (no CPU fallback exists)")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, U32, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint32, ctypes.c_size_t
    PP = ctypes.POINTER(ctypes.c_void_p)
    IP = ctypes.POINTER(ctypes.c_int)
    DP = ctypes.POINTER(goldy_gemm_desc)
    sig = {
        "goldy_abi_version": ([], I),
        "goldy_last_error": ([], ctypes.c_char_p),
        "goldy_variant_count": ([], I),
        "goldy_variant_info_get": ([I, ctypes.POINTER(goldy_variant_info)], I),
        "goldy_lut_load": ([ctypes.c_char_p, PP], I),
        "goldy_lut_from_memory": ([P, SZ, PP], I),
        "goldy_lut_free": ([P], None),
        "goldy_bucket_key": ([DP, ctypes.POINTER(U32)], I),
        "goldy_plan": ([DP, I, P, I, PP], I),
        "goldy_plan_ex": ([DP, I, P, P, I, PP], I),
        "goldy_predictor_load": ([ctypes.c_char_p, PP], I),
        "goldy_predictor_from_memory": ([P, SZ, PP], I),
        "goldy_predictor_free": ([P], None),
        "goldy_lut_lookup": ([P, DP, IP, IP], I),
        "goldy_lr_features": ([DP, P, I, ctypes.POINTER(ctypes.c_double)], I),
        "goldy_predict_cd": ([P, P, DP, IP, ctypes.POINTER(ctypes.c_double)], I),
        "goldy_schedule_build": ([DP, I, IP, IP, IP, I, PP], I),
        "goldy_schedule_query": ([P, IP, IP, IP, ctypes.POINTER(SZ)], I),
        "goldy_schedule_entry": ([P, I, IP, IP, IP, IP], I),
        "goldy_schedule_serialize": ([P, P, SZ, ctypes.POINTER(SZ)], I),
        "goldy_schedule_free": ([P], None),
        "goldy_run": ([P, PP, PP, PP, P, SZ, PP, I], I),
        "goldy_graph_create": ([P, PP, PP, PP, P, SZ, PP, I, PP], I),
        "goldy_run_ex": ([P, PP, PP, PP, P, SZ, PP, I, ctypes.POINTER(goldy_run_opts)], I),
        "goldy_graph_create_ex": ([P, PP, PP, PP, P, SZ, PP, I, ctypes.POINTER(goldy_run_opts), PP], I),
        "goldy_graph_launch": ([P, P], I),
        "goldy_exec_create": ([P, PP, PP, PP, P, SZ, PP, I, ctypes.POINTER(goldy_run_opts), PP], I),
        "goldy_exec_launch": ([P], I),
        "goldy_exec_time": ([PP, I, I, I, ctypes.POINTER(ctypes.c_float)], I),
        "goldy_partition_create": ([I, I, PP], I),
        "goldy_corun_plan": ([DP, ctypes.POINTER(goldy_ewise_desc), P, I, PP], I),
        "goldy_corun_query": ([P, IP, IP, IP, ctypes.POINTER(SZ)], I),
        "goldy_corun_run": ([P, P, P, P, P, SZ, P, P, P, PP, I], I),
        "goldy_corun_exec_create": ([P, P, P, P, P, SZ, P, P, P, PP, I, PP], I),
        "goldy_corun_free": ([P], None),
        "goldy_ewise_add": ([P, P, P, ctypes.c_int64, I, I, P], I),
        "goldy_partition_query": ([P, IP, PP, I], I),
        "goldy_partition_free": ([P], None),
        "goldy_exec_free": ([P], None),
        "goldy_graph_free": ([P], None),
        "goldy_gemm_noalloc": ([DP, I, P, P, P, P], I),
        "goldy_device_error": ([IP, I], I),
        "goldy_device_info": ([I, IP, IP], I),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


_lib = _load()


def _check(status: int, where: str) -> None:
    if status != GOLDY_OK:
        raise GoldyError(status, where, _lib.goldy_last_error().decode())


def _ptrs(values: Sequence[int]):
    arr = (ctypes.c_void_p * max(1, len(values)))()
    for i, v in enumerate(values):
        arr[i] = int(v) if v else None
    return arr


def _descs(descs: Sequence[goldy_gemm_desc]):
    arr = (goldy_gemm_desc * max(1, len(descs)))()
    for i, d in enumerate(descs):
        arr[i] = d
    return arr


def desc(M: int, N: int, K: int, c_dtype: int = GOLDY_F32, lda: Optional[int] = None,
         ldb: Optional[int] = None, ldc: Optional[int] = None, batch: int = 1, stride_a: Optional[int] = None,
         stride_b: Optional[int] = None, stride_c: Optional[int] = None) -> goldy_gemm_desc:
    """Descriptor of C (M x N) = A (M x K, row-major) * B (K x N, row-major),
    or of `batch` such products with entries packed back to back (default
    strides M*lda, K*ldb, M*ldc)."""
    lda = K if lda is None else lda
    ldb = N if ldb is None else ldb
    ldc = N if ldc is None else ldc
    return goldy_gemm_desc(M, N, K, lda, ldb, ldc, 0, 0, GOLDY_BF16, GOLDY_BF16, int(c_dtype), 0, int(batch),
                           M * lda if stride_a is None else stride_a, K * ldb if stride_b is None else stride_b,
                           M * ldc if stride_c is None else stride_c)


class _Handle:
    _free = None

    def __init__(self, ptr: ctypes.c_void_p):
        self.ptr = ptr

    def close(self) -> None:
        if self.ptr:
            type(self)._free(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Lut(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_lut_free(p))


class Predictor(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_predictor_free(p))


class Schedule(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_schedule_free(p))


class Graph(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_graph_free(p))


class Corun(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_corun_free(p))


class Partition(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_partition_free(p))


class Exec(_Handle):
    _free = staticmethod(lambda p: _lib.goldy_exec_free(p))


def goldy_abi_version() -> int:
    return int(_lib.goldy_abi_version())


def goldy_last_error() -> str:
    return _lib.goldy_last_error().decode()


def goldy_variant_count() -> int:
    return int(_lib.goldy_variant_count())


def goldy_variant_info_get(variant_id: int) -> dict:
    info = goldy_variant_info()
    _check(_lib.goldy_variant_info_get(int(variant_id), ctypes.byref(info)), "goldy_variant_info_get")
    return info.as_dict()


def goldy_lut_load(path: str = DEFAULT_LUT) -> Lut:
    out = ctypes.c_void_p()
    _check(_lib.goldy_lut_load(path.encode(), ctypes.byref(out)), "goldy_lut_load")
    return Lut(out)


def goldy_lut_from_memory(data: bytes) -> Lut:
    out = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(bytes(data), len(data))
    _check(_lib.goldy_lut_from_memory(buf, len(data), ctypes.byref(out)), "goldy_lut_from_memory")
    return Lut(out)


def goldy_bucket_key(d: goldy_gemm_desc) -> int:
    key = ctypes.c_uint32()
    _check(_lib.goldy_bucket_key(ctypes.byref(d), ctypes.byref(key)), "goldy_bucket_key")
    return int(key.value)


def goldy_plan(descs: Sequence[goldy_gemm_desc], lut: Lut, flags: int = GOLDY_PLAN_AUTO) -> Schedule:
    out = ctypes.c_void_p()
    _check(_lib.goldy_plan(_descs(descs), len(descs), lut.ptr if lut else None, int(flags),
                           ctypes.byref(out)), "goldy_plan")
    return Schedule(out)


def goldy_plan_ex(descs: Sequence[goldy_gemm_desc], lut: Lut, predictor: Optional[Predictor],
                  flags: int = GOLDY_PLAN_AUTO) -> Schedule:
    out = ctypes.c_void_p()
    _check(_lib.goldy_plan_ex(_descs(descs), len(descs), lut.ptr if lut else None,
                              predictor.ptr if predictor else None, int(flags), ctypes.byref(out)), "goldy_plan_ex")
    return Schedule(out)


def goldy_predictor_load(path: str = DEFAULT_PREDICTOR) -> Predictor:
    out = ctypes.c_void_p()
    _check(_lib.goldy_predictor_load(path.encode(), ctypes.byref(out)), "goldy_predictor_load")
    return Predictor(out)


def goldy_predictor_from_memory(data: bytes) -> Predictor:
    out = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(bytes(data), len(data))
    _check(_lib.goldy_predictor_from_memory(buf, len(data), ctypes.byref(out)), "goldy_predictor_from_memory")
    return Predictor(out)


def goldy_lut_lookup(lut: Lut, d: goldy_gemm_desc) -> Tuple[int, List[int]]:
    pref = ctypes.c_int()
    vs = (ctypes.c_int * 5)()
    _check(_lib.goldy_lut_lookup(lut.ptr, ctypes.byref(d), ctypes.byref(pref), vs), "goldy_lut_lookup")
    return pref.value, list(vs)


def goldy_lr_features(d: goldy_gemm_desc, lut: Lut, sm_count: int) -> List[float]:
    out = (ctypes.c_double * LR_FEATURES)()
    _check(_lib.goldy_lr_features(ctypes.byref(d), lut.ptr, int(sm_count), out), "goldy_lr_features")
    return list(out)


def goldy_predict_cd(p: Predictor, lut: Lut, d: goldy_gemm_desc) -> Tuple[int, List[float]]:
    cd = ctypes.c_int()
    probs = (ctypes.c_double * 5)()
    _check(_lib.goldy_predict_cd(p.ptr, lut.ptr, ctypes.byref(d), ctypes.byref(cd), probs), "goldy_predict_cd")
    return cd.value, list(probs)


def goldy_schedule_build(descs: Sequence[goldy_gemm_desc], group_of: Sequence[int],
                         variant_of: Sequence[int], slot_of: Sequence[int], flags: int = 0) -> Schedule:
    n = len(descs)
    IA = ctypes.c_int * max(1, n)
    out = ctypes.c_void_p()
    _check(_lib.goldy_schedule_build(_descs(descs), n, IA(*group_of), IA(*variant_of), IA(*slot_of),
                                     int(flags), ctypes.byref(out)), "goldy_schedule_build")
    return Schedule(out)


def goldy_schedule_query(s: Schedule) -> Tuple[int, int, int, int]:
    """(n_gemms, n_groups, max_streams, workspace_bytes)."""
    a, b, c, w = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_size_t()
    _check(_lib.goldy_schedule_query(s.ptr, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c),
                                     ctypes.byref(w)), "goldy_schedule_query")
    return a.value, b.value, c.value, int(w.value)


def goldy_schedule_entry(s: Schedule, gemm: int) -> Tuple[int, int, int, int]:
    """(group, variant, slot, cd) of GEMM ``gemm``."""
    g, v, sl, cd = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(_lib.goldy_schedule_entry(s.ptr, int(gemm), ctypes.byref(g), ctypes.byref(v),
                                     ctypes.byref(sl), ctypes.byref(cd)), "goldy_schedule_entry")
    return g.value, v.value, sl.value, cd.value


def goldy_schedule_serialize(s: Schedule) -> bytes:
    size = ctypes.c_size_t()
    _lib.goldy_schedule_serialize(s.ptr, None, 0, ctypes.byref(size))
    buf = ctypes.create_string_buffer(size.value)
    _check(_lib.goldy_schedule_serialize(s.ptr, buf, size.value, ctypes.byref(size)),
           "goldy_schedule_serialize")
    return buf.raw[:size.value]


def goldy_run(s: Schedule, A: Sequence[int], B: Sequence[int], C: Sequence[int], workspace: int,
              workspace_bytes: int, streams: Sequence[int]) -> None:
    _check(_lib.goldy_run(s.ptr, _ptrs(A), _ptrs(B), _ptrs(C), int(workspace) or None,
                          int(workspace_bytes), _ptrs(streams), len(streams)), "goldy_run")


def goldy_graph_create(s: Schedule, A: Sequence[int], B: Sequence[int], C: Sequence[int],
                       workspace: int, workspace_bytes: int, streams: Sequence[int]) -> Graph:
    out = ctypes.c_void_p()
    _check(_lib.goldy_graph_create(s.ptr, _ptrs(A), _ptrs(B), _ptrs(C), int(workspace) or None,
                                   int(workspace_bytes), _ptrs(streams), len(streams),
                                   ctypes.byref(out)), "goldy_graph_create")
    return Graph(out)


def _opts(ev_begin: Optional[Sequence[int]], ev_end: Optional[Sequence[int]], trace: int = 0,
          trace_ctas: int = 0, serial_launch: bool = False, inputs_ready: bool = False,
          wait_limit_us: int = 0, test_stall_first_stage: bool = False):
    o = goldy_run_opts()
    o.trace = int(trace) or None
    o.trace_ctas = int(trace_ctas)
    o.serial_launch = 1 if serial_launch else 0
    o.inputs_ready = 1 if inputs_ready else 0
    o.wait_limit_us = int(wait_limit_us)
    o.test_stall_first_stage = 1 if test_stall_first_stage else 0
    keep = []
    if ev_begin is not None:
        arr = _ptrs(ev_begin)
        keep.append(arr)
        o.ev_begin = ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))
    if ev_end is not None:
        arr = _ptrs(ev_end)
        keep.append(arr)
        o.ev_end = ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))
    return o, keep


def goldy_run_ex(s: Schedule, A: Sequence[int], B: Sequence[int], C: Sequence[int], workspace: int,
                 workspace_bytes: int, streams: Sequence[int], ev_begin: Optional[Sequence[int]] = None,
                 ev_end: Optional[Sequence[int]] = None, trace: int = 0, trace_ctas: int = 0,
                 serial_launch: bool = False, inputs_ready: bool = False, wait_limit_us: int = 0,
                 test_stall_first_stage: bool = False) -> None:
    """goldy_run with per-GEMM timing events (cudaEvent_t handles as ints),
    an optional device phase-trace buffer, the launch mode, early operand
    loads, the bounded-wait limit and the test stall hook (see
    goldy_run_opts)."""
    o, _keep = _opts(ev_begin, ev_end, trace, trace_ctas, serial_launch, inputs_ready, wait_limit_us,
                     test_stall_first_stage)
    _check(_lib.goldy_run_ex(s.ptr, _ptrs(A), _ptrs(B), _ptrs(C), int(workspace) or None,
                             int(workspace_bytes), _ptrs(streams), len(streams), ctypes.byref(o)),
           "goldy_run_ex")


def goldy_graph_create_ex(s: Schedule, A: Sequence[int], B: Sequence[int], C: Sequence[int],
                          workspace: int, workspace_bytes: int, streams: Sequence[int],
                          ev_begin: Optional[Sequence[int]] = None,
                          ev_end: Optional[Sequence[int]] = None, serial_launch: bool = False,
                          inputs_ready: bool = False) -> Graph:
    o, _keep = _opts(ev_begin, ev_end, serial_launch=serial_launch, inputs_ready=inputs_ready)
    out = ctypes.c_void_p()
    _check(_lib.goldy_graph_create_ex(s.ptr, _ptrs(A), _ptrs(B), _ptrs(C), int(workspace) or None,
                                      int(workspace_bytes), _ptrs(streams), len(streams),
                                      ctypes.byref(o), ctypes.byref(out)), "goldy_graph_create_ex")
    return Graph(out)


def goldy_exec_create(s: Schedule, A: Sequence[int], B: Sequence[int], C: Sequence[int], workspace: int,
                      workspace_bytes: int, streams: Sequence[int], ev_begin: Optional[Sequence[int]] = None,
                      ev_end: Optional[Sequence[int]] = None, trace: int = 0, trace_ctas: int = 0,
                      serial_launch: bool = False, inputs_ready: bool = False, wait_limit_us: int = 0) -> Exec:
    o, _keep = _opts(ev_begin, ev_end, trace, trace_ctas, serial_launch, inputs_ready, wait_limit_us)
    out = ctypes.c_void_p()
    _check(_lib.goldy_exec_create(s.ptr, _ptrs(A), _ptrs(B), _ptrs(C), int(workspace) or None,
                                  int(workspace_bytes), _ptrs(streams), len(streams), ctypes.byref(o),
                                  ctypes.byref(out)), "goldy_exec_create")
    return Exec(out)


def goldy_exec_time(execs: Sequence[Exec], warmup: int, reps: int) -> float:
    """Milliseconds per replay (see include/goldy.h)."""
    arr = (ctypes.c_void_p * len(execs))(*[e.ptr for e in execs])
    ms = ctypes.c_float()
    _check(_lib.goldy_exec_time(arr, len(execs), int(warmup), int(reps), ctypes.byref(ms)), "goldy_exec_time")
    return ms.value


def goldy_corun_plan(gemm: goldy_gemm_desc, n: int, dtype: int, lut: Lut, policy: int = GOLDY_PLAN_AUTO) -> Corun:
    """A GEMM co-scheduled with the element-wise add Z = X + Y of n elements."""
    ew = goldy_ewise_desc(int(n), int(dtype), 0)
    out = ctypes.c_void_p()
    _check(_lib.goldy_corun_plan(ctypes.byref(gemm), ctypes.byref(ew), lut.ptr if lut else None, int(policy),
                                 ctypes.byref(out)), "goldy_corun_plan")
    return Corun(out)


def goldy_corun_query(c: Corun) -> Tuple[int, int, int, int]:
    """(concurrent, gemm variant, add grid-cap divisor, workspace bytes)."""
    cc, v, rc, ws = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_size_t()
    _check(_lib.goldy_corun_query(c.ptr, ctypes.byref(cc), ctypes.byref(v), ctypes.byref(rc), ctypes.byref(ws)),
           "goldy_corun_query")
    return cc.value, v.value, rc.value, ws.value


def goldy_corun_run(c: Corun, A: int, B: int, C: int, workspace: int, workspace_bytes: int, X: int, Y: int, Z: int,
                    streams: Sequence[int]) -> None:
    _check(_lib.goldy_corun_run(c.ptr, A or None, B or None, C or None, workspace or None, int(workspace_bytes),
                                X or None, Y or None, Z or None, _ptrs(streams), len(streams)), "goldy_corun_run")


def goldy_corun_exec_create(c: Corun, A: int, B: int, C: int, workspace: int, workspace_bytes: int, X: int, Y: int,
                            Z: int, streams: Sequence[int]) -> "Exec":
    out = ctypes.c_void_p()
    _check(_lib.goldy_corun_exec_create(c.ptr, A or None, B or None, C or None, workspace or None,
                                        int(workspace_bytes), X or None, Y or None, Z or None, _ptrs(streams),
                                        len(streams), ctypes.byref(out)), "goldy_corun_exec_create")
    return Exec(out)


def goldy_ewise_add(X: int, Y: int, Z: int, n: int, dtype: int, rc_div: int, stream: int) -> None:
    _check(_lib.goldy_ewise_add(X or None, Y or None, Z or None, int(n), int(dtype), int(rc_div), stream or None),
           "goldy_ewise_add")


def goldy_partition_create(min_sms: int, n_streams: int = 16) -> Partition:
    out = ctypes.c_void_p()
    _check(_lib.goldy_partition_create(int(min_sms), int(n_streams), ctypes.byref(out)), "goldy_partition_create")
    return Partition(out)


def goldy_partition_query(p: Partition, n: int = 0) -> Tuple[int, List[int]]:
    """(SM count, the first n stream handles as integers)."""
    sm = ctypes.c_int()
    arr = (ctypes.c_void_p * max(1, n))()
    _check(_lib.goldy_partition_query(p.ptr, ctypes.byref(sm), arr, int(n)), "goldy_partition_query")
    return sm.value, [int(arr[k] or 0) for k in range(n)]


def goldy_exec_launch(e: Exec) -> None:
    _check(_lib.goldy_exec_launch(e.ptr), "goldy_exec_launch")


def goldy_graph_launch(g: Graph, stream: int) -> None:
    _check(_lib.goldy_graph_launch(g.ptr, int(stream) or None), "goldy_graph_launch")


def goldy_gemm_noalloc(d: goldy_gemm_desc, variant: int, A: int, B: int, C: int, stream: int = 0) -> None:
    """One GEMM with the library's compiled-in split-K scratch (no device
    allocation anywhere); see goldy.h for who needs it and its limits."""
    _check(_lib.goldy_gemm_noalloc(ctypes.byref(d), int(variant), int(A) or None, int(B) or None,
                                   int(C) or None, int(stream) or None), "goldy_gemm_noalloc")


def goldy_device_error(clear: bool = True) -> int:
    code = ctypes.c_int()
    _check(_lib.goldy_device_error(ctypes.byref(code), 1 if clear else 0), "goldy_device_error")
    return code.value


def goldy_device_info(variant_id: int = 0) -> Tuple[int, int]:
    """(SM count, resident CTAs per SM of the variant's kernel)."""
    sm, ctas = ctypes.c_int(), ctypes.c_int()
    _check(_lib.goldy_device_info(int(variant_id), ctypes.byref(sm), ctypes.byref(ctas)),
           "goldy_device_info")
    return sm.value, ctas.value


_SPLITS = (1, 2, 4, 8)
_RC_DIVS = (1, 2, 4)


def variant_id(kind: int, split: int, rc_div: int) -> int:
    """Variant id of (kind, split-K factor, grid-cap divisor): the registry's
    numbering (kind * 4 + split index) * 3 + RC index, checked against it."""
    if split not in _SPLITS or rc_div not in _RC_DIVS:
        raise KeyError((kind, split, rc_div))
    v = (int(kind) * 4 + _SPLITS.index(split)) * 3 + _RC_DIVS.index(rc_div)
    if not 0 <= v < goldy_variant_count():
        raise KeyError((kind, split, rc_div))
    info = goldy_variant_info_get(v)
    if info["kind"] != kind or info["rc_div"] != rc_div or info["split_k"] not in (split, 1):
        raise KeyError((kind, split, rc_div))
    return v


def kind_names() -> List[str]:
    names = {}
    for v in range(goldy_variant_count()):
        info = goldy_variant_info_get(v)
        names.setdefault(info["kind"], info["name"].split("_s")[0])
    return [names[k] for k in sorted(names)]

// Launch manager: runs a schedule on caller-owned streams.
//
// The paper's command processor dispatches the chosen GEMMs from their queue
// heads, as many at once as the predicted concurrency degree allows
// (Sec. 4.4).  Here each group of the schedule forks from streams[0] with an
// event, launches its GEMMs round-robin onto the group's stream slots (so at
// most CD GEMMs are in flight, each stream running its GEMMs back to back),
// and joins back into streams[0] before the next group starts.  In the fused
// launch mode the GEMMs of a wave that share a kernel kind go out as one
// persistent launch over all their tiles instead.  The whole run can be
// captured once into a CUDA graph and replayed with one launch.
//
// Per GEMM the host encodes two TMA tensor maps (A and B), sizes the
// persistent grid as min(units, resident CTAs per SM * SMs / rc_div) — the
// variant's resource constraint — and launches the kind's kernel.  Nothing
// here allocates device memory or synchronises.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "go_kernel.cuh"
#include "goldy_internal.h"

namespace goldy {

__device__ int g_device_error;   // kernels' error word (first failure wins)

struct Runtime {
  int device = -1;
  void* green = nullptr;   // green context the events were created under (null: the device's own)
  cudaEvent_t fork = nullptr;
  cudaEvent_t join[GOLDY_MAX_STREAMS] = {};
  cudaEvent_t started = nullptr;   // launch completion of a fused run's lead launch
};

void runtime_release(Runtime* rt) {
  if (!rt) return;
  if (rt->fork) cudaEventDestroy(rt->fork);
  if (rt->started) cudaEventDestroy(rt->started);
  for (cudaEvent_t e : rt->join)
    if (e) cudaEventDestroy(e);
  delete rt;
}

// Launch priority value meaning "none": the launch takes its stream's priority.
constexpr int kNoPriority = 1 << 30;

// One enqueued operation of a run.  goldy_run_ex executes them as it goes;
// goldy_exec_create records them (with copies of the kernel parameter blocks)
// so goldy_exec_launch can replay the run with plain launch calls.
struct Op {
  enum Kind { kKernel, kMemset2D, kEventRecord, kEventRecordExternal, kWait } kind = kKernel;
  cudaStream_t stream = nullptr;
  const void* fn = nullptr;
  unsigned grid = 0;
  unsigned block = 0;
  size_t smem = 0;
  int cluster = 0;
  bool pdl = false;                  // programmatic dependency on the previous kernel of the stream
  int prio = kNoPriority;            // launch priority (kNoPriority: the stream's)
  cudaEvent_t started = nullptr;     // launch-completion event to trigger (null: none)
  std::vector<uint64_t> params;      // 8-byte-aligned copy of the parameter block
  void* ptr = nullptr;
  size_t pitch = 0, width = 0, height = 0;
  cudaEvent_t ev = nullptr;
};

namespace {
thread_local std::vector<Op>* t_rec = nullptr;   // non-null: record instead of enqueue
// GO-Kernel launches carry a programmatic dependency on the previous kernel of
// their stream (the kernels wait for it before touching global memory) unless
// the run asks for serial launches
thread_local bool t_pdl = true;
// Run options copied into every launch's parameters (goldy_run_opts):
// early operand loads, the bounded-wait limit, and the test stall hook
// (first launch of the run only).
thread_local int32_t t_early = 0;
thread_local uint64_t t_wait_ns = 0;
thread_local int32_t t_stall = 0;
// Launch priority of the next GO-Kernel launch (kNoPriority: the stream's).
// A heterogeneous fused wave ranks its launches by work so the block
// scheduler hands SMs to the largest first and the others fill its tail.
thread_local int t_prio = kNoPriority;
// Event the next GO-Kernel launch triggers once all of its CTAs have begun
// (null: none); see the lead launch of a fused run in run_impl.
thread_local cudaEvent_t t_started = nullptr;
}

namespace {

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool init = false;
  int sm_count = 0;
  int prio_least = 0, prio_greatest = 0;    // cudaDeviceGetStreamPriorityRange
  int* err_word = nullptr;
  int ctas_per_sm[kNumKinds][2][2] = {};   // [kind][bf16 out][fused]; 0 = not yet set up
  int cluster_ok[kNumKinds][2][2][4] = {};  // [..][log2 cluster size]; 0 unknown, 1 yes, -1 no
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

goldy_status cuda_fail(cudaError_t e, const char* what) {
  return fail(GOLDY_ERR_CUDA, std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")");
}

const void* kernel_fn(int kind, int out_bf16, int fused) {
  switch (kind) {
    case 0: return kernel_fn_k0(out_bf16, fused);
    case 1: return kernel_fn_k1(out_bf16, fused);
    case 2: return kernel_fn_k2(out_bf16, fused);
    case 3: return kernel_fn_k3(out_bf16, fused);
    case 4: return kernel_fn_k4(out_bf16, fused);
    case 5: return kernel_fn_k5(out_bf16, fused);
    case 6: return kernel_fn_k6(out_bf16, fused);
    case 7: return kernel_fn_k7(out_bf16, fused);
    case 8: return kernel_fn_k8(out_bf16, fused);
    case 9: return kernel_fn_k9(out_bf16, fused);
    case 10: return kernel_fn_k10(out_bf16, fused);
    default: return nullptr;
  }
}

// Per-device setup: SM count, error word address, encode entry point.
goldy_status device_state(DeviceState** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(GOLDY_ERR_UNSUPPORTED, "device index too large");
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceState& d = g_dev[dev];
  if (!d.init) {
    e = cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    e = cudaDeviceGetStreamPriorityRange(&d.prio_least, &d.prio_greatest);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetStreamPriorityRange");
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.err_word), g_device_error);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress");
    if (!g_encode) {
      cudaDriverEntryPointQueryResult q;
      void* fn = nullptr;
      e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
      if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
        return fail(GOLDY_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    d.init = true;
  }
  *out = &d;
  return GOLDY_OK;
}

// Resident CTAs per SM of one kernel (kind, dtype, launch form) on this
// device; also opts the kernel into its dynamic shared-memory size the first
// time.
goldy_status kernel_setup(DeviceState& d, int kind, int out_bf16, int fused, int* ctas) {
  std::lock_guard<std::mutex> lock(g_mu);
  int& c = d.ctas_per_sm[kind][out_bf16][fused];
  if (c == 0) {
    const void* fn = kernel_fn(kind, out_bf16, fused);
    if (!fn) return fail(GOLDY_ERR_UNSUPPORTED, "no kernel for this kind");
    const KindInfo& k = kKinds[kind];
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes(k));
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute");
    int occ = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, kThreads, smem_bytes(k));
    if (e != cudaSuccess) return cuda_fail(e, "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
    // tensor memory is not part of the occupancy query: 512 columns per SM
    occ = std::min(occ, 512 / tmem_cols(k));
    if (occ < 1) return fail(GOLDY_ERR_UNSUPPORTED, "kernel does not fit on an SM");
    c = occ;
  }
  *ctas = c;
  return GOLDY_OK;
}

// Launch `fn` with one parameter block; as clusters of `cluster` CTAs when
// cluster > 1.
cudaError_t launch_kernel_now(const void* fn, unsigned grid, size_t smem, cudaStream_t stream, void* params,
                              int cluster, unsigned block = kThreads, bool pdl = false, int prio = kNoPriority,
                              cudaEvent_t started = nullptr) {
  void* args[] = {params};
  if (cluster <= 1 && !pdl && prio == kNoPriority && !started)
    return cudaLaunchKernel(fn, dim3(grid), dim3(block), args, smem, stream);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[4];
  unsigned n = 0;
  if (started) {
    attr[n].id = cudaLaunchAttributeLaunchCompletionEvent;
    attr[n].val.launchCompletionEvent.event = started;
    attr[n].val.launchCompletionEvent.flags = 0;
    ++n;
  }
  if (prio != kNoPriority) {
    attr[n].id = cudaLaunchAttributePriority;
    attr[n].val.priority = prio;
    ++n;
  }
  if (cluster > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = unsigned(cluster);
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelExC(&cfg, fn, args);
}

// A GO-Kernel launch (recorded when t_rec is set).
cudaError_t launch_kernel(const void* fn, unsigned grid, size_t smem, cudaStream_t stream, const void* params,
                          size_t params_size, int cluster) {
  if (!t_rec)
    return launch_kernel_now(fn, grid, smem, stream, const_cast<void*>(params), cluster, kThreads, t_pdl, t_prio,
                             t_started);
  Op op;
  op.kind = Op::kKernel;
  op.stream = stream;
  op.fn = fn;
  op.grid = grid;
  op.smem = smem;
  op.cluster = cluster;
  op.pdl = t_pdl;
  op.prio = t_prio;
  op.started = t_started;
  op.params.resize((params_size + 7) / 8);
  std::memcpy(op.params.data(), params, params_size);
  t_rec->push_back(std::move(op));
  return cudaSuccess;
}

// A kernel with `block` threads per CTA and no cluster (recorded like launch_kernel).
cudaError_t launch_kernel_threads(const void* fn, unsigned grid, unsigned block, size_t smem, cudaStream_t stream,
                                  const void* params, size_t params_size) {
  if (!t_rec) return launch_kernel_now(fn, grid, smem, stream, const_cast<void*>(params), 0, block);
  Op op;
  op.kind = Op::kKernel;
  op.stream = stream;
  op.fn = fn;
  op.grid = grid;
  op.block = block;
  op.smem = smem;
  op.params.resize((params_size + 7) / 8);
  std::memcpy(op.params.data(), params, params_size);
  t_rec->push_back(std::move(op));
  return cudaSuccess;
}

cudaError_t enq_memset2d(void* ptr, size_t pitch, size_t width, size_t height, cudaStream_t stream) {
  if (!t_rec) return cudaMemset2DAsync(ptr, pitch, 0, width, height, stream);
  Op op;
  op.kind = Op::kMemset2D;
  op.stream = stream;
  op.ptr = ptr;
  op.pitch = pitch;
  op.width = width;
  op.height = height;
  t_rec->push_back(std::move(op));
  return cudaSuccess;
}

cudaError_t enq_event_record(cudaEvent_t ev, cudaStream_t stream, bool external = false) {
  if (!t_rec) {
    if (!external) return cudaEventRecord(ev, stream);
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(stream, &cs);
    if (e != cudaSuccess) return e;
    return cudaEventRecordWithFlags(ev, stream, cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : 0);
  }
  Op op;
  op.kind = external ? Op::kEventRecordExternal : Op::kEventRecord;
  op.stream = stream;
  op.ev = ev;
  t_rec->push_back(std::move(op));
  return cudaSuccess;
}

cudaError_t enq_wait(cudaStream_t stream, cudaEvent_t ev) {
  if (!t_rec) return cudaStreamWaitEvent(stream, ev, 0);
  Op op;
  op.kind = Op::kWait;
  op.stream = stream;
  op.ev = ev;
  t_rec->push_back(std::move(op));
  return cudaSuccess;
}

cudaError_t replay(const Op& op) {
  switch (op.kind) {
    case Op::kKernel:
      return launch_kernel_now(op.fn, op.grid, op.smem, op.stream, const_cast<uint64_t*>(op.params.data()),
                               op.cluster, op.block ? op.block : kThreads, op.pdl, op.prio, op.started);
    case Op::kMemset2D: return cudaMemset2DAsync(op.ptr, op.pitch, 0, op.width, op.height, op.stream);
    case Op::kEventRecord: return cudaEventRecord(op.ev, op.stream);
    case Op::kEventRecordExternal: return cudaEventRecordWithFlags(op.ev, op.stream, 0);
    case Op::kWait: return cudaStreamWaitEvent(op.stream, op.ev, 0);
  }
  return cudaErrorInvalidValue;
}

// Can clusters of `cluster` CTAs of this kernel be resident at all?
bool cluster_feasible(DeviceState& d, int kind, int out_bf16, int fused, int cluster) {
  const int li = cluster == 2 ? 1 : cluster == 4 ? 2 : cluster == 8 ? 3 : 0;
  if (li == 0) return false;
  std::lock_guard<std::mutex> lock(g_mu);
  int& c = d.cluster_ok[kind][out_bf16][fused][li];
  if (c == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(cluster));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = size_t(smem_bytes(kKinds[kind]));
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = unsigned(cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&n, kernel_fn(kind, out_bf16, fused), &cfg);
    c = (e == cudaSuccess && n > 0) ? 1 : -1;
    if (e != cudaSuccess) cudaGetLastError();     // clear; fall back to the unclustered reduction
  }
  return c > 0;
}

// Grid of a launch: the persistent cap, and a whole number of clusters.
unsigned launch_grid(int64_t units, int64_t cap, int cluster) {
  int64_t g = std::min<int64_t>(units, cap);
  if (cluster > 1) g = std::max<int64_t>(cluster, (g / cluster) * cluster);
  return unsigned(g);
}

// Pair kinds: every unit (a 256-row tile) occupies a cluster of two CTAs.
unsigned pair_grid(int64_t units, int64_t cap) {
  const int64_t pairs = std::max<int64_t>(1, std::min<int64_t>(units, cap / 2));
  return unsigned(2 * pairs);
}

// Tensor map of a (batch x outer x inner) array: rows of `row_bytes`, batch
// entries `batch_bytes` apart; boxes of box_outer rows x box_inner elements
// of one entry, 128-byte swizzled.
goldy_status encode_3d(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint64_t batch,
                       uint64_t row_bytes, uint64_t batch_bytes, uint32_t box_inner, uint32_t box_outer,
                       CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  cuuint64_t dims[3] = {inner, outer, batch};
  cuuint64_t strides[2] = {row_bytes, batch_bytes};
  cuuint32_t box[3] = {box_inner, box_outer, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(m, dtype, 3, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuTensorMapEncodeTiled failed with code " + std::to_string(int(r)));
  return GOLDY_OK;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// One GEMM's slot of a launch: tensor maps and work description.
template <int MAXG>
goldy_status fill_slot(LaunchParams<MAXG>& p, int j, const GemmPlan& gp, const void* A, const void* B, void* C,
                       uint8_t* ws, int32_t unit_begin) {
  const goldy_gemm_desc& g = gp.desc;
  const KindInfo& k = kKinds[gp.kind];
  // batch strides in bytes; a single GEMM gets the packed stride (never read)
  const bool batched = g.batch > 1;
  const uint64_t sa = uint64_t(batched ? g.stride_a : g.M * g.lda) * 2;
  const uint64_t sb = uint64_t(batched ? g.stride_b : g.K * g.ldb) * 2;
  goldy_status st = encode_3d(&p.tmap_a[j], A, uint64_t(g.K), uint64_t(g.M), uint64_t(g.batch), uint64_t(g.lda) * 2,
                              sa, kBlockK, uint32_t(a_box_rows(k)));
  if (st != GOLDY_OK) return st;
  st = encode_3d(&p.tmap_b[j], B, uint64_t(g.N), uint64_t(g.K), uint64_t(g.batch), uint64_t(g.ldb) * 2, sb, 64,
                 kBlockK);
  if (st != GOLDY_OK) return st;
  GemmWork& w = p.g[j];
  w.c = C;
  w.ldc = g.ldc;
  w.batch = int32_t(g.batch);
  w.c_bstride = batched ? g.stride_c : g.M * g.ldc;
  w.m = int32_t(g.M);
  w.n = int32_t(g.N);
  w.k = int32_t(g.K);
  w.tiles_m = int32_t(gp.tiles_m);
  w.tiles_n = int32_t(gp.tiles_n);
  w.split = gp.split;
  w.k_blocks = int32_t(gp.k_blocks);
  w.unit_begin = unit_begin;
  // C through TMA stores: kinds that keep staging buffers, 16-byte aligned C
  // and rows; the epilogue writes 128-byte rows (32 fp32 / 64 bf16 columns)
  const size_t es = g.c_dtype == GOLDY_BF16 ? 2 : 4;
  // (kinds with a whole SM store every tile this way; the two-per-SM kinds,
  // which keep no staging buffers, only a CTA's last tile, staged in its
  // idle operand ring)
  w.c_tma = 0;
  const uint64_t sc = uint64_t(w.c_bstride) * es;
  if (!k.swap_ab && gp.split == 1 && aligned(C, 16) && (size_t(g.ldc) * es) % 16 == 0 && sc % 16 == 0) {
    st = encode_3d(&p.tmap_c[j], C, uint64_t(g.N), uint64_t(g.M), uint64_t(g.batch), uint64_t(g.ldc) * es, sc,
                   uint32_t(128 / es), 128,
                   g.c_dtype == GOLDY_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32);
    if (st != GOLDY_OK) return st;
    w.c_tma = 1;
  }
  if (gp.split > 1) {
    w.ws_part = reinterpret_cast<float*>(ws + gp.ws_part_off);
    w.ws_cnt = reinterpret_cast<uint32_t*>(ws + gp.ws_cnt_off);
  }
  return GOLDY_OK;
}

// GEMMs that need no kernel: nothing to write (M or N is 0) or C = 0 (K is 0).
bool degenerate(const GemmPlan& gp) { return gp.desc.M == 0 || gp.desc.N == 0 || gp.desc.K == 0; }

goldy_status launch_degenerate(const GemmPlan& gp, void* C, cudaStream_t stream) {
  const goldy_gemm_desc& g = gp.desc;
  if (g.M == 0 || g.N == 0) return GOLDY_OK;
  const size_t es = g.c_dtype == GOLDY_BF16 ? 2 : 4;
  const int64_t cstride = g.batch > 1 ? g.stride_c : g.M * g.ldc;
  if (cstride == g.M * g.ldc) {   // entries packed: one 2-D fill over all of them
    cudaError_t e = enq_memset2d(C, size_t(g.ldc) * es, size_t(g.N) * es, size_t(g.M * g.batch), stream);
    return e == cudaSuccess ? GOLDY_OK : cuda_fail(e, "cudaMemset2DAsync");
  }
  for (int64_t b = 0; b < g.batch; ++b) {
    cudaError_t e = enq_memset2d(static_cast<char*>(C) + size_t(b * cstride) * es, size_t(g.ldc) * es,
                                 size_t(g.N) * es, size_t(g.M), stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemset2DAsync");
  }
  return GOLDY_OK;
}

// ---------------------------------------------------------------------------
// SM partitions (CUDA green contexts).  A partition is a green context owning
// a subset of the SMs; work on its streams runs on those SMs only.  Every
// entry point that enqueues work makes the partition of its first stream
// current for the duration of the call and sizes grids for its SM count.
// ---------------------------------------------------------------------------
struct GreenApi {
  PFN_cuDeviceGet_v2000 device_get = nullptr;
  PFN_cuDeviceGetDevResource_v12040 dev_resource = nullptr;
  PFN_cuDevSmResourceSplitByCount_v12040 split = nullptr;
  PFN_cuDevResourceGenerateDesc_v12040 gen_desc = nullptr;
  PFN_cuGreenCtxCreate_v12040 create = nullptr;
  PFN_cuGreenCtxDestroy_v12040 destroy = nullptr;
  PFN_cuGreenCtxGetDevResource_v12040 ctx_resource = nullptr;
  PFN_cuGreenCtxStreamCreate_v12050 stream_create = nullptr;
  PFN_cuStreamDestroy_v4000 stream_destroy = nullptr;
  PFN_cuStreamGetGreenCtx_v12040 stream_green = nullptr;
  PFN_cuCtxFromGreenCtx_v12040 to_ctx = nullptr;
  PFN_cuCtxPushCurrent_v4000 push = nullptr;
  PFN_cuCtxPopCurrent_v4000 pop = nullptr;
  bool ok = false;
};

const GreenApi& green_api() {
  static GreenApi api = [] {
    GreenApi a;
    auto get = [](const char* name, int ver, void** fn) {
      cudaDriverEntryPointQueryResult q;
      return cudaGetDriverEntryPointByVersion(name, fn, ver, cudaEnableDefault, &q) == cudaSuccess &&
             q == cudaDriverEntryPointSuccess && *fn;
    };
    bool ok = true;
    ok &= get("cuDeviceGet", 2000, reinterpret_cast<void**>(&a.device_get));
    ok &= get("cuDeviceGetDevResource", 12040, reinterpret_cast<void**>(&a.dev_resource));
    ok &= get("cuDevSmResourceSplitByCount", 12040, reinterpret_cast<void**>(&a.split));
    ok &= get("cuDevResourceGenerateDesc", 12040, reinterpret_cast<void**>(&a.gen_desc));
    ok &= get("cuGreenCtxCreate", 12040, reinterpret_cast<void**>(&a.create));
    ok &= get("cuGreenCtxDestroy", 12040, reinterpret_cast<void**>(&a.destroy));
    ok &= get("cuGreenCtxGetDevResource", 12040, reinterpret_cast<void**>(&a.ctx_resource));
    ok &= get("cuGreenCtxStreamCreate", 12050, reinterpret_cast<void**>(&a.stream_create));
    ok &= get("cuStreamDestroy", 4000, reinterpret_cast<void**>(&a.stream_destroy));
    ok &= get("cuStreamGetGreenCtx", 12040, reinterpret_cast<void**>(&a.stream_green));
    ok &= get("cuCtxFromGreenCtx", 12040, reinterpret_cast<void**>(&a.to_ctx));
    ok &= get("cuCtxPushCurrent", 4000, reinterpret_cast<void**>(&a.push));
    ok &= get("cuCtxPopCurrent", 4000, reinterpret_cast<void**>(&a.pop));
    a.ok = ok;
    return a;
  }();
  return api;
}

// SMs the current run may use: the partition's when its streams belong to a
// green context, else the device's (0).
thread_local int t_sms = 0;

// Makes the green context of `stream` (if it has one) current on this thread
// until destroyed, and sets t_sms to its SM count.
class PartitionScope {
 public:
  goldy_status enter(void* stream) {
    green_ = nullptr;
    if (!stream) return GOLDY_OK;
    const GreenApi& g = green_api();
    if (!g.ok) return GOLDY_OK;                  // no green contexts: every stream is the device's
    CUgreenCtx gc = nullptr;
    if (g.stream_green(static_cast<CUstream>(stream), &gc) != CUDA_SUCCESS || !gc) return GOLDY_OK;
    CUcontext ctx = nullptr;
    if (g.to_ctx(&ctx, gc) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuCtxFromGreenCtx failed");
    CUdevResource res;
    std::memset(&res, 0, sizeof(res));
    if (g.ctx_resource(gc, &res, CU_DEV_RESOURCE_TYPE_SM) != CUDA_SUCCESS)
      return fail(GOLDY_ERR_CUDA, "cuGreenCtxGetDevResource failed");
    if (g.push(ctx) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuCtxPushCurrent failed");
    green_ = gc;
    saved_sms_ = t_sms;
    t_sms = int(res.sm.smCount);
    return GOLDY_OK;
  }
  void* green() const { return green_; }
  ~PartitionScope() {
    if (!green_) return;
    CUcontext popped = nullptr;
    green_api().pop(&popped);
    t_sms = saved_sms_;
  }

 private:
  void* green_ = nullptr;
  int saved_sms_ = 0;
};
int sms(const DeviceState& d) { return t_sms > 0 ? std::min(t_sms, d.sm_count) : d.sm_count; }

// Phase-trace buffer of the current goldy_run_ex call (null: off).
thread_local unsigned long long* t_trace = nullptr;
thread_local size_t t_trace_ctas = 0;
thread_local size_t t_trace_used = 0;   // CTAs of the run's earlier launches

// The launches of one run trace into consecutive regions of the buffer, in
// launch order; a launch that does not fit in what is left is not traced.
unsigned long long* trace_for(unsigned grid) {
  if (!t_trace || t_trace_used + grid > t_trace_ctas) return nullptr;
  unsigned long long* region = t_trace + t_trace_used * 16;
  t_trace_used += grid;
  return region;
}

// scale > 0: the launch's grid cap is its variant's cap times `scale` (set for
// heterogeneous fused waves, see goldy_run_ex), at most the whole GPU.
goldy_status launch_gemm(DeviceState& d, const GemmPlan& gp, const void* A, const void* B, void* C, uint8_t* ws,
                         cudaStream_t stream, double scale = 0.0) {
  if (degenerate(gp)) return launch_degenerate(gp, C, stream);
  const KindInfo& k = kKinds[gp.kind];
  const int out_bf16 = gp.desc.c_dtype == GOLDY_BF16 ? 1 : 0;
  int ctas = 0;
  goldy_status st = kernel_setup(d, gp.kind, out_bf16, 0, &ctas);
  if (st != GOLDY_OK) return st;
  if (gp.units > int64_t(1) << 30) return fail(GOLDY_ERR_UNSUPPORTED, "too many tiles in one GEMM");

  LaunchParams<1> p;
  std::memset(&p, 0, sizeof(p));
  st = fill_slot(p, 0, gp, A, B, C, ws, 0);
  if (st != GOLDY_OK) return st;
  p.n_gemms = 1;
  p.total_units = int32_t(gp.units);
  p.err = d.err_word;
  p.wait_ns = t_wait_ns;
  p.early_loads = t_early;
  p.stall_test = t_stall;
  t_stall = 0;

  const Variant v = variant_of(gp.variant);
  int64_t cap = std::max<int64_t>(1, int64_t(ctas) * sms(d) / v.rc_div);
  if (scale > 0.0) cap = std::min<int64_t>(int64_t(ctas) * sms(d), std::max<int64_t>(1, int64_t(double(cap) * scale)));
  if (k.pair) {
    const unsigned grid = pair_grid(gp.units, cap);
    p.trace = trace_for(grid);
    cudaError_t e =
        launch_kernel(kernel_fn(gp.kind, out_bf16, 0), grid, size_t(smem_bytes(k)), stream, &p, sizeof(p), 2);
    if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernel (pair)");
    return GOLDY_OK;
  }
  const int cluster = (gp.split > 1 && cluster_feasible(d, gp.kind, out_bf16, 0, gp.split)) ? gp.split : 0;
  p.cluster = cluster;
  const unsigned grid = launch_grid(gp.units, cap, cluster);
  p.trace = trace_for(grid);
  cudaError_t e =
      launch_kernel(kernel_fn(gp.kind, out_bf16, 0), grid, size_t(smem_bytes(k)), stream, &p, sizeof(p), cluster);
  if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernel");
  return GOLDY_OK;
}

// One launch over the tiles of `count` (<= kMaxFused) GEMMs of one kind and
// output dtype.  The grid cap is the sum of the members' own caps (each
// GO-Kernel keeps the share of the GPU it was tuned for), at most the whole
// GPU.
goldy_status launch_fused(DeviceState& d, const goldy_schedule* s, const int* members_in, int count,
                          const void* const* A, const void* const* B, void* const* C, uint8_t* ws,
                          cudaStream_t stream, double scale = 0.0) {
  const GemmPlan& g0 = s->gemms[members_in[0]];
  const KindInfo& k = kKinds[g0.kind];
  const int out_bf16 = g0.desc.c_dtype == GOLDY_BF16 ? 1 : 0;
  int ctas = 0;
  goldy_status st = kernel_setup(d, g0.kind, out_bf16, 1, &ctas);
  if (st != GOLDY_OK) return st;
  static thread_local LaunchParams<kMaxFused> p;   // ~5 KB: keep it off the stack
  std::memset(&p, 0, sizeof(p));
  int64_t units = 0, cap = 0;
  // clusters need one split factor for every GEMM of the launch
  int split = g0.split;
  for (int j = 0; j < count; ++j) {
    const GemmPlan& gp = s->gemms[members_in[j]];
    units += gp.units;
    cap += std::max<int64_t>(1, int64_t(ctas) * sms(d) / variant_of(gp.variant).rc_div);
    if (gp.split != split) split = 0;
  }
  if (units > int64_t(1) << 30) return fail(GOLDY_ERR_UNSUPPORTED, "too many tiles in one launch");
  if (scale > 0.0) cap = std::max<int64_t>(1, int64_t(double(cap) * scale));
  cap = std::min<int64_t>(cap, int64_t(ctas) * sms(d));
  const int cluster = (!k.pair && split > 1 && cluster_feasible(d, g0.kind, out_bf16, 1, split)) ? split : 0;
  const unsigned grid = k.pair ? pair_grid(units, cap) : launch_grid(units, cap, cluster);
  // Units handed out by a counter (longest first) instead of round-robin:
  // when the CTAs take several units each and the GEMMs' units differ in
  // length (2x or more), a static order leaves the launch's end to the CTAs
  // that drew the long ones (a launch of 868 six-K-block units and 15
  // 93-K-block units: 123.6 -> 111.5 us for its set).  Equal units gain
  // nothing and pay the counter (eight equal GEMMs: 17.9 -> 19.4 us).  Not
  // with cluster-reduced split-K (a cluster's CTAs take the splits of one
  // tile together) nor the pair kernel.
  int members[kMaxFused];
  for (int j = 0; j < count; ++j) members[j] = members_in[j];
  auto unit_len = [&](int i) { return int64_t(s->gemms[i].k_blocks) / std::max(1, s->gemms[i].split); };
  int64_t shortest = INT64_MAX, longest = 0;
  for (int j = 0; j < count; ++j) {
    shortest = std::min(shortest, unit_len(members[j]));
    longest = std::max(longest, unit_len(members[j]));
  }
  bool dyn = !k.pair && cluster == 0 && units > int64_t(grid) && ws != nullptr && longest >= 2 * shortest;
  for (int j = 0; j < count && dyn; ++j) dyn = s->gemms[members[j]].ws_dyn_off != ~size_t(0);
  if (dyn)
    std::stable_sort(members, members + count, [&](int a, int b) { return unit_len(a) > unit_len(b); });
  units = 0;
  for (int j = 0; j < count; ++j) {
    const GemmPlan& gp = s->gemms[members[j]];
    st = fill_slot(p, j, gp, A[members[j]], B[members[j]], C[members[j]], ws, int32_t(units));
    if (st != GOLDY_OK) return st;
    units += gp.units;
  }
  p.n_gemms = count;
  p.total_units = int32_t(units);
  p.err = d.err_word;
  p.wait_ns = t_wait_ns;
  p.early_loads = t_early;
  p.stall_test = t_stall;
  t_stall = 0;
  p.dyn = dyn ? reinterpret_cast<uint32_t*>(ws + s->gemms[members[0]].ws_dyn_off) : nullptr;
  p.trace = trace_for(grid);
  if (k.pair) {
    cudaError_t e =
        launch_kernel(kernel_fn(g0.kind, out_bf16, 1), grid, size_t(smem_bytes(k)), stream, &p, sizeof(p), 2);
    if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernel (fused pair)");
    return GOLDY_OK;
  }
  p.cluster = cluster;
  cudaError_t e =
      launch_kernel(kernel_fn(g0.kind, out_bf16, 1), grid, size_t(smem_bytes(k)), stream, &p, sizeof(p), cluster);
  if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernel (fused)");
  return GOLDY_OK;
}

}  // namespace
}  // namespace goldy

using namespace goldy;

namespace {
// Record a caller's timing event on `stream`; inside a capture it must be an
// external record to become a real node of the graph.
cudaError_t record_hook(void* ev, cudaStream_t stream) {
  if (!ev) return cudaSuccess;
  return enq_event_record(static_cast<cudaEvent_t>(ev), stream, true);
}
}  // namespace

extern "C" goldy_status goldy_run(const goldy_schedule* s, const void* const* A, const void* const* B,
                                  void* const* C, void* workspace, size_t workspace_bytes, void* const* streams,
                                  int n_streams) {
  return goldy_run_ex(s, A, B, C, workspace, workspace_bytes, streams, n_streams, nullptr);
}

namespace goldy {
Runtime* new_runtime(int dev, void* green, goldy_status* st) {
  Runtime* rt = new Runtime();
  rt->device = dev;
  rt->green = green;
  cudaError_t e = cudaEventCreateWithFlags(&rt->fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&rt->started, cudaEventDisableTiming);
  for (int k = 0; k < GOLDY_MAX_STREAMS && e == cudaSuccess; ++k)
    e = cudaEventCreateWithFlags(&rt->join[k], cudaEventDisableTiming);
  if (e != cudaSuccess) {
    runtime_release(rt);
    *st = cuda_fail(e, "cudaEventCreate");
    return nullptr;
  }
  *st = GOLDY_OK;
  return rt;
}
}  // namespace goldy

namespace {
// Restores the per-run thread-local launch options when a run ends, on every
// return path, so that no option of one run leaks into another entry point.
struct RunOptionsReset {
  ~RunOptionsReset() {
    t_trace = nullptr;
    t_trace_ctas = 0;
    t_trace_used = 0;
    t_pdl = true;
    t_early = 0;
    t_wait_ns = 0;
    t_stall = 0;
  }
};
}  // namespace

// The run itself; `own_rt`, if given, supplies the fork/join events (a
// recorded run owns its events), otherwise the schedule's are used.
static goldy_status run_impl(const goldy_schedule* s, const void* const* A, const void* const* B, void* const* C,
                             void* workspace, size_t workspace_bytes, void* const* streams, int n_streams,
                             const goldy_run_opts* opts, Runtime* own_rt) {
  if (!s || !A || !B || !C || !streams) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  if (n_streams < s->max_streams) return fail(GOLDY_ERR_INVALID_ARG, "fewer streams than the schedule needs");
  if (s->workspace_bytes > 0) {
    if (!workspace || workspace_bytes < s->workspace_bytes)
      return fail(GOLDY_ERR_INVALID_ARG, "workspace missing or smaller than goldy_schedule_query reports");
    if (!aligned(workspace, 256)) return fail(GOLDY_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  }
  for (size_t i = 0; i < s->gemms.size(); ++i) {
    const goldy_gemm_desc& g = s->gemms[i].desc;
    if (g.M == 0 || g.N == 0) continue;
    const size_t es = g.c_dtype == GOLDY_BF16 ? 2 : 4;
    if (!C[i] || !aligned(C[i], es)) return fail(GOLDY_ERR_INVALID_ARG, "gemm " + std::to_string(i) + ": C null or misaligned");
    if (g.K == 0) continue;
    if (!A[i] || !B[i] || !aligned(A[i], 16) || !aligned(B[i], 16))
      return fail(GOLDY_ERR_INVALID_ARG, "gemm " + std::to_string(i) + ": A and B must be 16-byte aligned device pointers");
  }
  DeviceState* d = nullptr;
  goldy_status st = device_state(&d);
  if (st != GOLDY_OK) return st;
  PartitionScope part;
  st = part.enter(streams[0]);
  if (st != GOLDY_OK) return st;

  Runtime* rt = own_rt;
  if (!rt) {
    goldy_schedule* ms = const_cast<goldy_schedule*>(s);
    int dev = 0;
    cudaGetDevice(&dev);
    if (ms->rt && (ms->rt->device != dev || ms->rt->green != part.green())) {
      runtime_release(ms->rt);
      ms->rt = nullptr;
    }
    if (!ms->rt) {
      ms->rt = new_runtime(dev, part.green(), &st);
      if (!ms->rt) return st;
    }
    rt = ms->rt;
  }
  cudaStream_t main = static_cast<cudaStream_t>(streams[0]);
  uint8_t* ws = static_cast<uint8_t*>(workspace);

  RunOptionsReset reset_options;
  t_trace = opts ? static_cast<unsigned long long*>(opts->trace) : nullptr;
  t_trace_ctas = opts ? opts->trace_ctas : 0;
  t_trace_used = 0;
  t_pdl = !(opts && opts->serial_launch);
  t_early = (opts && opts->inputs_ready) ? 1 : 0;
  t_wait_ns = opts ? uint64_t(opts->wait_limit_us) * 1000ull : 0;
  t_stall = (opts && opts->test_stall_first_stage) ? 1 : 0;
  auto hook = [&](void* const* evs, const int* members, int n, cudaStream_t stream) -> goldy_status {
    if (!evs) return GOLDY_OK;
    for (int j = 0; j < n; ++j) {
      cudaError_t e = record_hook(evs[members[j]], stream);
      if (e != cudaSuccess) return cuda_fail(e, "timing event");
    }
    return GOLDY_OK;
  };
  const bool fused = (s->flags & GOLDY_PLAN_FUSED) != 0;

  // Launch sets.  Streams mode: one per GEMM, on the GEMM's slot.  Fused
  // mode: a group's members taken CD at a time form waves; in a wave, the
  // GEMMs of one kind and output dtype share a launch on the slot of the
  // first of them.
  struct LaunchSet {
    int group, slot, n, degenerate, wave;
    double scale;     // grid-cap scale for heterogeneous fused waves (0: none)
    int rank;         // rank by FLOPs among the launches of its wave (0: largest)
    int prio;         // launch priority (kNoPriority: the stream's)
    double flops;
    int members[kMaxFused];
  };
  std::vector<LaunchSet> sets;
  sets.reserve(s->gemms.size());
  for (size_t g = 0; g < s->groups.size(); ++g) {
    const Group& grp = s->groups[g];
    const int size = int(grp.members.size());
    const int wave = fused ? std::max(1, grp.cd) : 1;
    for (int w0 = 0; w0 < size; w0 += wave) {
      const size_t first_set = sets.size();
      for (int j = w0; j < std::min(size, w0 + wave); ++j) {
        const int i = grp.members[j];
        const GemmPlan& gp = s->gemms[i];
        size_t target = sets.size();
        if (fused && !degenerate(gp))
          for (size_t t = first_set; t < sets.size(); ++t) {
            const GemmPlan& g0 = s->gemms[sets[t].members[0]];
            if (!sets[t].degenerate && sets[t].n < kMaxFused && g0.kind == gp.kind &&
                g0.desc.c_dtype == gp.desc.c_dtype) {
              target = t;
              break;
            }
          }
        if (target == sets.size()) {
          LaunchSet ls{};
          ls.group = int(g);
          ls.slot = gp.slot;
          ls.degenerate = degenerate(gp) ? 1 : 0;
          ls.wave = w0;
          ls.prio = kNoPriority;
          sets.push_back(ls);
        }
        sets[target].members[sets[target].n++] = i;
        sets[target].flops += 2.0 * double(gp.desc.M) * double(gp.desc.N) * double(gp.desc.K) *
                              double(std::max<int64_t>(1, gp.desc.batch));
      }
    }
  }
  // Priority levels from the device's greatest (level 0) to its least.
  const int prio_step = d->prio_greatest <= d->prio_least ? 1 : -1;
  const int prio_levels = std::abs(d->prio_least - d->prio_greatest) + 1;
  auto level = [&](int lv) { return d->prio_greatest + prio_step * std::min(lv, prio_levels - 1); };
  // A fused wave whose GEMMs are of different kinds runs one launch per
  // kind, side by side.  A GO-Kernel tuned for CD c was sized as one of c
  // co-runners sharing the GPU; a launch that carries m of the wave's c GEMMs
  // therefore gets c/m times its members' caps (at most the whole GPU), and
  // the wave's launches are ranked by FLOPs into launch priorities, so the
  // largest gets the SMs first and smaller ones fill the SMs it frees in its
  // tail.
  const bool soft_groups = fused && s->groups.size() > 1;
  if (fused) {
    for (size_t t0 = 0; t0 < sets.size();) {
      size_t t1 = t0;
      int kernels = 0, wave_size = 0;
      while (t1 < sets.size() && sets[t1].group == sets[t0].group && sets[t1].wave == sets[t0].wave) {
        wave_size += sets[t1].n;
        if (!sets[t1].degenerate) ++kernels;
        ++t1;
      }
      // A plan of one group whose wave fits on the GPU unscaled: the scale is
      // bounded by the largest uniform one (at most c/m) at which its launches
      // are all resident at once, since over-subscribing left the
      // lower-priority launch of a small wave waiting for SMs (a two-GEMM
      // set: 14.4 -> 10.5 us with the bound).
      // Plans of several groups keep the full c/m: there the same bound
      // measured 5-28% slower (the over-subscribed first group's CTAs take
      // SMs as they free up, ahead of the later groups' launches).
      double fit = 1e30;
      if (kernels > 1 && !soft_groups) {
        struct Need {
          double units, cap, ctas;   // CTAs of work, the launch's own cap, CTAs per SM
        };
        std::vector<Need> need;
        for (size_t t = t0; t < t1; ++t) {
          if (sets[t].degenerate) continue;
          const GemmPlan& g0 = s->gemms[sets[t].members[0]];
          int ctas = 0;
          st = kernel_setup(*d, g0.kind, g0.desc.c_dtype == GOLDY_BF16 ? 1 : 0, sets[t].n > 1 ? 1 : 0, &ctas);
          if (st != GOLDY_OK) return st;
          Need nd{0.0, 0.0, double(ctas)};
          for (int j = 0; j < sets[t].n; ++j) {
            const GemmPlan& gp = s->gemms[sets[t].members[j]];
            nd.units += double(gp.units) * (kKinds[gp.kind].pair ? 2.0 : 1.0);
            nd.cap += std::max(1.0, double(ctas) * sms(*d) / variant_of(gp.variant).rc_div);
          }
          need.push_back(nd);
        }
        auto sm_use = [&](double sc) {
          double u = 0.0;
          for (const Need& nd : need) u += std::min(nd.units, std::min(nd.cap * sc, nd.ctas * sms(*d))) / nd.ctas;
          return u;
        };
        // (a wave that over-subscribes the GPU unscaled keeps c/m: its smaller
        // launches run in the largest one's tail, where a quarter-GPU cap
        // left one at two rounds — 160 -> 194 us on a four-GEMM set)
        if (sm_use(1.0) <= double(sms(*d))) {
          double lo = 1.0, hi = double(wave_size);
          if (sm_use(hi) <= double(sms(*d))) lo = hi;
          for (int it = 0; it < 30 && hi - lo > 1e-3; ++it) {
            const double mid = 0.5 * (lo + hi);
            (sm_use(mid) <= double(sms(*d)) ? lo : hi) = mid;
          }
          fit = lo;
        }
      }
      for (size_t t = t0; t < t1; ++t) {
        if (sets[t].degenerate) continue;
        for (size_t u = t0; u < t1; ++u)
          if (u != t && !sets[u].degenerate &&
              (sets[u].flops > sets[t].flops || (sets[u].flops == sets[t].flops && u < t)))
            ++sets[t].rank;
        if (kernels > 1) {
          sets[t].scale = std::min(double(wave_size) / double(sets[t].n), std::max(1.0, fit));
          sets[t].prio = level(sets[t].rank);
        }
        // groups of a fused plan are not separated by a join: group g's
        // launches rank g levels below the first group's, so a later group
        // fills the SMs an earlier group frees in its tail
        if (soft_groups) sets[t].prio = level(sets[t].group + sets[t].rank);
      }
      t0 = t1;
    }
  }
  // Fork the side streams from streams[0] and join them back: around each
  // group in streams mode (groups run one after another), once around the
  // whole run in fused mode.
  auto fork = [&](uint32_t side) -> goldy_status {
    if (!side) return GOLDY_OK;
    cudaError_t e = enq_event_record(rt->fork, main);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    for (int k = 1; k < GOLDY_MAX_STREAMS; ++k)
      if (side >> k & 1) {
        e = enq_wait(static_cast<cudaStream_t>(streams[k]), rt->fork);
        if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
      }
    return GOLDY_OK;
  };
  auto join = [&](uint32_t side) -> goldy_status {
    for (int k = 1; k < GOLDY_MAX_STREAMS; ++k)
      if (side >> k & 1) {
        cudaError_t e = enq_event_record(rt->join[k], static_cast<cudaStream_t>(streams[k]));
        if (e == cudaSuccess) e = enq_wait(main, rt->join[k]);
        if (e != cudaSuccess) return cuda_fail(e, "join event");
      }
    return GOLDY_OK;
  };
  // Fused mode: when the first wave has several launches, its largest (the
  // lead) goes out first and triggers rt->started once all of its CTAs have
  // begun; every other stream waits for that before its first launch.
  // Priorities alone do not order the start: CTAs of a single-CTA kernel take
  // SMs one at a time as the previous run's CTAs leave, while a cluster of
  // the pair kernel needs two neighbouring SMs free at once, so a smaller
  // launch used to occupy the GPU first.  (The event is best effort: the
  // others may start later, never before the lead has begun.  Inside a stream
  // capture the graph edge it becomes waited for the whole lead kernel —
  // hetero_pair replayed 54 -> 63 us — so captured runs go without it.)
  size_t lead = sets.size();
  cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
  if (fused && !t_rec) {
    cudaError_t e = cudaStreamIsCapturing(main, &capturing);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamIsCapturing");
  }
  if (fused && capturing == cudaStreamCaptureStatusNone) {
    int kernels = 0;
    for (size_t t = 0; t < sets.size() && sets[t].group == 0 && sets[t].wave == 0; ++t)
      if (!sets[t].degenerate) {
        ++kernels;
        if (sets[t].rank == 0) lead = t;
      }
    // only a pair-kernel lead needs it (its clusters need two free SMs at
    // once); for single-CTA launches the priorities suffice, and the event
    // and waits measured ~4 us on a two-GEMM set of small kernels
    if (kernels < 2 || (lead < sets.size() && !kKinds[s->gemms[sets[lead].members[0]].kind].pair)) lead = sets.size();
  }
  // Fused runs with inputs_ready go out on streams[0] alone, largest launch
  // of each wave first: each launch's loads and MMAs start in the previous
  // one's tail (programmatic dependent launch), with no fork or join, and
  // consecutive runs overlap the same way; each launch's epilogue waits for
  // the previous kernel only where it first writes global memory.  Measured
  // over the 64 randomized sets, back to back: with runs of at most 5
  // launches on one stream and the rest on the CD streams, roofline
  // fraction geomean 0.443 (tensor-bound 0.556); with every run on one
  // stream 0.446 (0.561), runs of 6-9 launches up to 13% faster, two of them
  // 5-8% slower.  (Before the epilogues waited only at their first global
  // write, runs of more than 5 launches measured 4-6% slower on one stream.)
  // Without inputs_ready a launch would wait for the previous one to
  // complete, so those runs keep the streams.
  int n_launches = 0;
  for (const LaunchSet& ls : sets) n_launches += ls.degenerate ? 0 : 1;
  const bool one_stream = fused && t_early && n_launches >= 2;
  if (one_stream) lead = sets.size();
  std::vector<size_t> order;
  order.reserve(sets.size());
  if (lead < sets.size()) order.push_back(lead);
  for (size_t t = 0; t < sets.size(); ++t)
    if (t != lead) order.push_back(t);
  if (one_stream)
    std::stable_sort(order.begin(), order.end(), [&](size_t a, size_t b) {
      if (sets[a].group != sets[b].group) return sets[a].group < sets[b].group;
      if (sets[a].wave != sets[b].wave) return sets[a].wave < sets[b].wave;
      return sets[a].rank < sets[b].rank;
    });
  const bool pdl = t_pdl;
  int last_group[GOLDY_MAX_STREAMS];
  bool waited[GOLDY_MAX_STREAMS];
  for (int k = 0; k < GOLDY_MAX_STREAMS; ++k) {
    last_group[k] = -1;
    waited[k] = false;
  }
  for (size_t t0 = 0; t0 < order.size();) {
    // the launches dispatched between one fork and its join
    size_t t1 = t0;
    while (t1 < order.size() && (fused || sets[order[t1]].group == sets[order[t0]].group)) ++t1;
    uint32_t used = 0;
    for (size_t t = t0; t < t1; ++t) used |= 1u << (one_stream ? 0 : sets[order[t]].slot);
    const uint32_t side = used & ~1u;            // slots other than 0 fork from and join into streams[0]
    st = fork(side);
    if (st != GOLDY_OK) return st;
    for (size_t t = t0; t < t1; ++t) {
      const LaunchSet& ls = sets[order[t]];
      cudaStream_t stream = static_cast<cudaStream_t>(streams[one_stream ? 0 : ls.slot]);
      if (lead < sets.size() && order[t] != lead && !waited[ls.slot] && ls.slot != sets[lead].slot) {
        cudaError_t e = enq_wait(stream, rt->started);
        if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent (lead started)");
        waited[ls.slot] = true;
      }
      st = hook(opts ? opts->ev_begin : nullptr, ls.members, ls.n, stream);
      if (st != GOLDY_OK) return st;
      // a kernel that follows another group's kernel on its stream starts
      // only once that kernel is done (no early set-up holding SMs)
      t_pdl = pdl && (one_stream || last_group[ls.slot] < 0 || last_group[ls.slot] == ls.group);
      last_group[ls.slot] = ls.group;
      t_prio = ls.prio;
      t_started = order[t] == lead ? rt->started : nullptr;
      if (ls.n == 1) {
        const int i = ls.members[0];
        st = launch_gemm(*d, s->gemms[i], A[i], B[i], C[i], ws, stream, ls.scale);
      } else {
        st = launch_fused(*d, s, ls.members, ls.n, A, B, C, ws, stream, ls.scale);
      }
      t_prio = kNoPriority;
      t_started = nullptr;
      t_pdl = pdl;
      if (st != GOLDY_OK) return st;
      st = hook(opts ? opts->ev_end : nullptr, ls.members, ls.n, stream);
      if (st != GOLDY_OK) return st;
    }
    st = join(side);
    if (st != GOLDY_OK) return st;
    t0 = t1;
  }
  return ok();
}

extern "C" goldy_status goldy_run_ex(const goldy_schedule* s, const void* const* A, const void* const* B,
                                     void* const* C, void* workspace, size_t workspace_bytes, void* const* streams,
                                     int n_streams, const goldy_run_opts* opts) {
  return run_impl(s, A, B, C, workspace, workspace_bytes, streams, n_streams, opts, nullptr);
}

struct goldy_exec {
  std::vector<Op> ops;
  Runtime* rt = nullptr;
  Runtime* rt2 = nullptr;    // a co-run's own fork/join events
  CUcontext ctx = nullptr;   // the partition's context to make current while replaying (null: none)
  cudaStream_t main = nullptr;
};

extern "C" goldy_status goldy_exec_create(const goldy_schedule* s, const void* const* A, const void* const* B,
                                          void* const* C, void* workspace, size_t workspace_bytes,
                                          void* const* streams, int n_streams, const goldy_run_opts* opts,
                                          goldy_exec** out) {
  if (!out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (!streams || n_streams < 1) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  PartitionScope part;
  goldy_status st = part.enter(streams[0]);
  if (st != GOLDY_OK) return st;
  goldy_exec* x = new (std::nothrow) goldy_exec();
  if (!x) return fail(GOLDY_ERR_NOMEM, "out of host memory");
  if (part.green() && green_api().to_ctx(&x->ctx, static_cast<CUgreenCtx>(part.green())) != CUDA_SUCCESS) {
    delete x;
    return fail(GOLDY_ERR_CUDA, "cuCtxFromGreenCtx failed");
  }
  x->main = static_cast<cudaStream_t>(streams[0]);
  x->rt = new_runtime(dev, part.green(), &st);
  if (!x->rt) {
    delete x;
    return st;
  }
  t_rec = &x->ops;
  st = run_impl(s, A, B, C, workspace, workspace_bytes, streams, n_streams, opts, x->rt);
  t_rec = nullptr;
  if (st != GOLDY_OK) {
    std::string why = goldy_last_error();
    runtime_release(x->rt);
    delete x;
    return fail(st, why);
  }
  *out = x;
  return ok();
}

extern "C" goldy_status goldy_exec_launch(const goldy_exec* x) {
  if (!x) return fail(GOLDY_ERR_INVALID_ARG, "null exec");
  if (x->ctx && green_api().push(x->ctx) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuCtxPushCurrent failed");
  cudaError_t e = cudaSuccess;
  for (const Op& op : x->ops) {
    e = replay(op);
    if (e != cudaSuccess) break;
  }
  if (x->ctx) {
    CUcontext popped = nullptr;
    green_api().pop(&popped);
  }
  if (e != cudaSuccess) return cuda_fail(e, "goldy_exec_launch");
  return ok();
}

extern "C" goldy_status goldy_exec_time(const goldy_exec* const* execs, int n, int warmup, int reps,
                                        float* ms_per_rep) {
  if (!execs || n < 1 || warmup < 0 || reps < 1 || !ms_per_rep) return fail(GOLDY_ERR_INVALID_ARG, "bad argument");
  for (int i = 0; i < n; ++i)
    if (!execs[i] || execs[i]->ctx != execs[0]->ctx || execs[i]->main != execs[0]->main)
      return fail(GOLDY_ERR_INVALID_ARG, "prepared runs must share their context and first stream");
  const goldy_exec* x0 = execs[0];
  if (x0->ctx && green_api().push(x0->ctx) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuCtxPushCurrent failed");
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  cudaError_t e = cudaEventCreate(&e0);
  if (e == cudaSuccess) e = cudaEventCreate(&e1);
  for (int k = 0; k < warmup && e == cudaSuccess; ++k)
    for (const Op& op : execs[k % n]->ops)
      if ((e = replay(op)) != cudaSuccess) break;
  if (e == cudaSuccess) e = cudaEventRecord(e0, x0->main);
  for (int k = 0; k < reps && e == cudaSuccess; ++k)
    for (const Op& op : execs[k % n]->ops)
      if ((e = replay(op)) != cudaSuccess) break;
  if (e == cudaSuccess) e = cudaEventRecord(e1, x0->main);
  if (e == cudaSuccess) e = cudaEventSynchronize(e1);
  float ms = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (x0->ctx) {
    CUcontext popped = nullptr;
    green_api().pop(&popped);
  }
  if (e != cudaSuccess) return cuda_fail(e, "goldy_exec_time");
  *ms_per_rep = ms / float(reps);
  return ok();
}

extern "C" void goldy_exec_free(goldy_exec* x) {
  if (!x) return;
  runtime_release(x->rt);
  runtime_release(x->rt2);
  delete x;
}

// ---------------------------------------------------------------------------
// Element-wise add and a GEMM co-scheduled with it
// ---------------------------------------------------------------------------
static goldy_status launch_ewise(const DeviceState& d, const goldy_ewise_desc& ew, const void* X, const void* Y,
                                 void* Z, int rc_div, cudaStream_t stream) {
  if (ew.n == 0) return GOLDY_OK;
  EwiseParams p;
  std::memset(&p, 0, sizeof(p));
  p.x = X;
  p.y = Y;
  p.z = Z;
  p.n = ew.n;
  p.vec_ok = (aligned(X, 16) && aligned(Y, 16) && aligned(Z, 16)) ? 1 : 0;
  const int64_t per_vec = ew.dtype == GOLDY_BF16 ? 8 : 4;
  const int64_t work = p.vec_ok ? (ew.n + per_vec - 1) / per_vec : ew.n;
  const int64_t cap = std::max<int64_t>(1, int64_t(kEwiseCtasPerSm) * sms(d) / rc_div);
  const unsigned grid = unsigned(std::max<int64_t>(1, std::min<int64_t>(cap, (work + kEwiseThreads - 1) / kEwiseThreads)));
  cudaError_t e = launch_kernel_threads(ewise_kernel_fn(ew.dtype == GOLDY_BF16 ? 1 : 0), grid, kEwiseThreads, 0,
                                        stream, &p, sizeof(p));
  if (e != cudaSuccess) return cuda_fail(e, "cudaLaunchKernel (element-wise add)");
  return GOLDY_OK;
}

static goldy_status check_ewise(const goldy_ewise_desc& ew, const void* X, const void* Y, void* Z, int rc_div) {
  if (ew.n < 0 || ew.reserved != 0 || (ew.dtype != GOLDY_BF16 && ew.dtype != GOLDY_F32))
    return fail(GOLDY_ERR_INVALID_ARG, "bad element-wise descriptor");
  if (rc_div != 1 && rc_div != 2 && rc_div != 4) return fail(GOLDY_ERR_INVALID_ARG, "rc_div must be 1, 2 or 4");
  const size_t es = ew.dtype == GOLDY_BF16 ? 2 : 4;
  if (ew.n > 0 && (!X || !Y || !Z || !aligned(X, es) || !aligned(Y, es) || !aligned(Z, es)))
    return fail(GOLDY_ERR_INVALID_ARG, "element-wise operands null or misaligned");
  return GOLDY_OK;
}

extern "C" goldy_status goldy_ewise_add(const void* X, const void* Y, void* Z, int64_t n, int dtype, int rc_div,
                                        void* stream) {
  goldy_ewise_desc ew{n, dtype, 0};
  goldy_status st = check_ewise(ew, X, Y, Z, rc_div);
  if (st != GOLDY_OK) return st;
  DeviceState* d = nullptr;
  st = device_state(&d);
  if (st != GOLDY_OK) return st;
  PartitionScope part;
  st = part.enter(stream);
  if (st != GOLDY_OK) return st;
  st = launch_ewise(*d, ew, X, Y, Z, rc_div, static_cast<cudaStream_t>(stream));
  return st == GOLDY_OK ? ok() : st;
}

// gemm_rt: events of the GEMM's run (null: the GEMM schedule's own);
// corun_rt: the fork/join events of the two streams (null: the co-run's own).
static goldy_status corun_impl(const goldy_corun* c, const void* A, const void* B, void* C, void* ws,
                               size_t ws_bytes, const void* X, const void* Y, void* Z, void* const* streams,
                               int n_streams, Runtime* gemm_rt, Runtime* corun_rt) {
  if (!c || !streams) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  if (n_streams < (c->concurrent ? 2 : 1)) return fail(GOLDY_ERR_INVALID_ARG, "fewer streams than the co-run needs");
  goldy_status st = check_ewise(c->ew, X, Y, Z, c->add_rc_div);
  if (st != GOLDY_OK) return st;
  DeviceState* d = nullptr;
  st = device_state(&d);
  if (st != GOLDY_OK) return st;
  PartitionScope part;
  st = part.enter(streams[0]);
  if (st != GOLDY_OK) return st;
  cudaStream_t s0 = static_cast<cudaStream_t>(streams[0]);
  const void* const a[1] = {A};
  const void* const b[1] = {B};
  void* const cc[1] = {C};
  if (!c->concurrent) {
    st = run_impl(c->gemm, a, b, cc, ws, ws_bytes, streams, 1, nullptr, gemm_rt);
    if (st != GOLDY_OK) return st;
    st = launch_ewise(*d, c->ew, X, Y, Z, c->add_rc_div, s0);
    return st == GOLDY_OK ? ok() : st;
  }
  Runtime* rt = corun_rt;
  if (!rt) {
    goldy_corun* mc = const_cast<goldy_corun*>(c);
    int dev = 0;
    cudaGetDevice(&dev);
    if (mc->rt && (mc->rt->device != dev || mc->rt->green != part.green())) {
      runtime_release(mc->rt);
      mc->rt = nullptr;
    }
    if (!mc->rt) {
      mc->rt = new_runtime(dev, part.green(), &st);
      if (!mc->rt) return st;
    }
    rt = mc->rt;
  }
  cudaStream_t s1 = static_cast<cudaStream_t>(streams[1]);
  cudaError_t e = enq_event_record(rt->fork, s0);
  if (e == cudaSuccess) e = enq_wait(s1, rt->fork);
  if (e != cudaSuccess) return cuda_fail(e, "co-run fork");
  st = run_impl(c->gemm, a, b, cc, ws, ws_bytes, streams, 1, nullptr, gemm_rt);
  if (st != GOLDY_OK) return st;
  st = launch_ewise(*d, c->ew, X, Y, Z, c->add_rc_div, s1);
  if (st != GOLDY_OK) return st;
  e = enq_event_record(rt->join[0], s1);
  if (e == cudaSuccess) e = enq_wait(s0, rt->join[0]);
  if (e != cudaSuccess) return cuda_fail(e, "co-run join");
  return ok();
}

extern "C" goldy_status goldy_corun_run(const goldy_corun* c, const void* A, const void* B, void* C, void* workspace,
                                        size_t workspace_bytes, const void* X, const void* Y, void* Z,
                                        void* const* streams, int n_streams) {
  return corun_impl(c, A, B, C, workspace, workspace_bytes, X, Y, Z, streams, n_streams, nullptr, nullptr);
}

extern "C" goldy_status goldy_corun_exec_create(const goldy_corun* c, const void* A, const void* B, void* C,
                                                void* workspace, size_t workspace_bytes, const void* X,
                                                const void* Y, void* Z, void* const* streams, int n_streams,
                                                goldy_exec** out) {
  if (!out || !c || !streams || n_streams < 1) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) return cuda_fail(ce, "cudaGetDevice");
  PartitionScope part;
  goldy_status st = part.enter(streams[0]);
  if (st != GOLDY_OK) return st;
  goldy_exec* x = new (std::nothrow) goldy_exec();
  if (!x) return fail(GOLDY_ERR_NOMEM, "out of host memory");
  if (part.green() && green_api().to_ctx(&x->ctx, static_cast<CUgreenCtx>(part.green())) != CUDA_SUCCESS) {
    delete x;
    return fail(GOLDY_ERR_CUDA, "cuCtxFromGreenCtx failed");
  }
  x->main = static_cast<cudaStream_t>(streams[0]);
  x->rt = new_runtime(dev, part.green(), &st);
  if (x->rt) x->rt2 = new_runtime(dev, part.green(), &st);
  if (!x->rt || !x->rt2) {
    goldy_exec_free(x);
    return st;
  }
  t_rec = &x->ops;
  st = corun_impl(c, A, B, C, workspace, workspace_bytes, X, Y, Z, streams, n_streams, x->rt, x->rt2);
  t_rec = nullptr;
  if (st != GOLDY_OK) {
    std::string why = goldy_last_error();
    goldy_exec_free(x);
    return fail(st, why);
  }
  *out = x;
  return ok();
}

struct goldy_graph {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
};

extern "C" goldy_status goldy_graph_create(const goldy_schedule* s, const void* const* A, const void* const* B,
                                           void* const* C, void* workspace, size_t workspace_bytes,
                                           void* const* streams, int n_streams, goldy_graph** out) {
  return goldy_graph_create_ex(s, A, B, C, workspace, workspace_bytes, streams, n_streams, nullptr, out);
}

extern "C" goldy_status goldy_graph_create_ex(const goldy_schedule* s, const void* const* A, const void* const* B,
                                              void* const* C, void* workspace, size_t workspace_bytes,
                                              void* const* streams, int n_streams, const goldy_run_opts* opts,
                                              goldy_graph** out) {
  if (!out || !streams) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  PartitionScope part;
  goldy_status pst = part.enter(streams[0]);
  if (pst != GOLDY_OK) return pst;
  cudaStream_t main = static_cast<cudaStream_t>(streams[0]);
  cudaError_t e = cudaStreamBeginCapture(main, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamBeginCapture");
  goldy_status st = goldy_run_ex(s, A, B, C, workspace, workspace_bytes, streams, n_streams, opts);
  std::string why = st == GOLDY_OK ? "" : goldy_last_error();
  cudaGraph_t graph = nullptr;
  e = cudaStreamEndCapture(main, &graph);
  if (st != GOLDY_OK) {
    if (graph) cudaGraphDestroy(graph);
    return fail(st, why);
  }
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamEndCapture");
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  if (e != cudaSuccess) {
    cudaGraphDestroy(graph);
    return cuda_fail(e, "cudaGraphInstantiate");
  }
  goldy_graph* g = new goldy_graph();
  g->graph = graph;
  g->exec = exec;
  *out = g;
  return ok();
}

extern "C" goldy_status goldy_graph_launch(const goldy_graph* g, void* stream) {
  if (!g) return fail(GOLDY_ERR_INVALID_ARG, "null graph");
  PartitionScope part;
  goldy_status pst = part.enter(stream);
  if (pst != GOLDY_OK) return pst;
  cudaError_t e = cudaGraphLaunch(g->exec, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphLaunch");
  return ok();
}

extern "C" void goldy_graph_free(goldy_graph* g) {
  if (!g) return;
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  delete g;
}

extern "C" goldy_status goldy_device_error(int* code, int clear) {
  if (!code) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  DeviceState* d = nullptr;
  goldy_status st = device_state(&d);
  if (st != GOLDY_OK) return st;
  cudaError_t e = cudaMemcpy(code, d->err_word, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy (error word)");
  if (clear && *code != 0) {
    const int zero = 0;
    e = cudaMemcpy(d->err_word, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy (clear error word)");
  }
  return ok();
}

extern "C" goldy_status goldy_device_info(int variant_id, int* sm_count, int* ctas_per_sm) {
  if (variant_id < 0 || variant_id >= kNumVariants) return fail(GOLDY_ERR_INVALID_ARG, "variant id out of range");
  DeviceState* d = nullptr;
  goldy_status st = device_state(&d);
  if (st != GOLDY_OK) return st;
  const Variant v = variant_of(variant_id);
  int ctas = 0;
  st = kernel_setup(*d, v.kind, 0, 0, &ctas);
  if (st != GOLDY_OK) return st;
  if (sm_count) *sm_count = d->sm_count;
  if (ctas_per_sm) *ctas_per_sm = ctas;
  return ok();
}

namespace goldy {
// Launch one GEMM whose plan fields (kind, tiles, split, workspace offsets)
// are already filled in, with `ws` as the workspace base, after zeroing
// `clear_bytes` bytes of it at `clear_off` on the same stream.  Shares the
// per-device setup and the launch code of goldy_run, and like goldy_run runs
// inside the SM partition `stream` belongs to (its green context current,
// grid caps from its SM count).
goldy_status launch_planned_gemm(const GemmPlan& gp, const void* A, const void* B, void* C, unsigned char* ws,
                                 void* stream, size_t clear_off, size_t clear_bytes) {
  DeviceState* d = nullptr;
  goldy_status st = device_state(&d);
  if (st != GOLDY_OK) return st;
  PartitionScope part;
  st = part.enter(stream);
  if (st != GOLDY_OK) return st;
  if (clear_bytes > 0) {
    cudaError_t e = cudaMemsetAsync(ws + clear_off, 0, clear_bytes, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync (split-K counters)");
  }
  return launch_gemm(*d, gp, A, B, C, ws, static_cast<cudaStream_t>(stream));
}
}  // namespace goldy

// ---------------------------------------------------------------------------
// SM partitions
// ---------------------------------------------------------------------------
struct goldy_partition {
  CUgreenCtx ctx = nullptr;
  int sm_count = 0;
  std::vector<CUstream> streams;
};

extern "C" void goldy_partition_free(goldy_partition* p) {
  if (!p) return;
  const GreenApi& g = green_api();
  for (CUstream st : p->streams)
    if (st) g.stream_destroy(st);
  if (p->ctx) g.destroy(p->ctx);
  delete p;
}

extern "C" goldy_status goldy_partition_create(int min_sms, int n_streams, goldy_partition** out) {
  if (!out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  if (n_streams < 1 || n_streams > GOLDY_MAX_STREAMS) return fail(GOLDY_ERR_INVALID_ARG, "stream count out of range");
  const GreenApi& g = green_api();
  if (!g.ok) return fail(GOLDY_ERR_UNSUPPORTED, "green contexts are not available from this driver");
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) return cuda_fail(ce, "cudaGetDevice");
  ce = cudaFree(nullptr);   // the primary context must exist before a green context retains it
  if (ce != cudaSuccess) return cuda_fail(ce, "cudaFree(0)");
  CUdevice cu = 0;
  if (g.device_get(&cu, dev) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuDeviceGet failed");
  CUdevResource all;
  std::memset(&all, 0, sizeof(all));
  if (g.dev_resource(cu, &all, CU_DEV_RESOURCE_TYPE_SM) != CUDA_SUCCESS)
    return fail(GOLDY_ERR_CUDA, "cuDeviceGetDevResource failed");
  CUdevResource part;
  std::memset(&part, 0, sizeof(part));
  if (min_sms <= 0 || unsigned(min_sms) >= all.sm.smCount) {
    part = all;                                   // the whole device, as a partition
  } else {
    unsigned groups = 1;
    CUdevResource rest;
    std::memset(&rest, 0, sizeof(rest));
    if (g.split(&part, &groups, &all, &rest, 0, unsigned(min_sms)) != CUDA_SUCCESS || groups != 1)
      return fail(GOLDY_ERR_UNSUPPORTED, "cannot split off a partition of " + std::to_string(min_sms) + " SMs");
  }
  CUdevResourceDesc desc = nullptr;
  if (g.gen_desc(&desc, &part, 1) != CUDA_SUCCESS) return fail(GOLDY_ERR_CUDA, "cuDevResourceGenerateDesc failed");
  goldy_partition* p = new (std::nothrow) goldy_partition();
  if (!p) return fail(GOLDY_ERR_NOMEM, "out of host memory");
  if (g.create(&p->ctx, desc, cu, CU_GREEN_CTX_DEFAULT_STREAM) != CUDA_SUCCESS) {
    p->ctx = nullptr;
    goldy_partition_free(p);
    return fail(GOLDY_ERR_CUDA, "cuGreenCtxCreate failed");
  }
  CUdevResource got;
  std::memset(&got, 0, sizeof(got));
  if (g.ctx_resource(p->ctx, &got, CU_DEV_RESOURCE_TYPE_SM) != CUDA_SUCCESS) {
    goldy_partition_free(p);
    return fail(GOLDY_ERR_CUDA, "cuGreenCtxGetDevResource failed");
  }
  p->sm_count = int(got.sm.smCount);
  p->streams.assign(size_t(n_streams), nullptr);
  for (int k = 0; k < n_streams; ++k) {
    if (g.stream_create(&p->streams[size_t(k)], p->ctx, CU_STREAM_NON_BLOCKING, 0) != CUDA_SUCCESS) {
      p->streams[size_t(k)] = nullptr;
      goldy_partition_free(p);
      return fail(GOLDY_ERR_CUDA, "cuGreenCtxStreamCreate failed");
    }
  }
  *out = p;
  return ok();
}

extern "C" goldy_status goldy_partition_query(const goldy_partition* p, int* sm_count, void** streams, int n) {
  if (!p) return fail(GOLDY_ERR_INVALID_ARG, "null partition");
  if (n < 0 || n > int(p->streams.size()) || (n > 0 && !streams))
    return fail(GOLDY_ERR_INVALID_ARG, "stream count out of range");
  if (sm_count) *sm_count = p->sm_count;
  for (int k = 0; k < n; ++k) streams[k] = p->streams[size_t(k)];
  return ok();
}

// goldy_gemm_noalloc: one GEMM through a GO-Kernel without any device
// allocation by the caller or by the library.
//
// Split-K GO-Kernels need scratch memory for their partial tiles and arrival
// counters; goldy_run takes it from a caller-supplied workspace.  Some callers
// cannot provide one because they are not allowed to allocate device memory
// where they run GEMMs: runtimes that give a kernel library a fixed memory
// budget and forbid further device allocations, plugins inside a host
// framework that owns every device allocation, and latency-critical paths
// where cudaMalloc's implicit synchronisation is not acceptable.  For them
// this entry point keeps the scratch in a fixed array compiled into the
// library.
//
// The array, g_noalloc_scratch, holds kNoAllocScratchBytes (32 MiB).  Every
// GPU that loads this library's device code holds one copy until the process
// exits.  A request whose scratch would exceed it is rejected with
// GOLDY_ERR_INVALID_ARG before anything is launched.
//
// In host code `g_noalloc_scratch` is only a host-side stand-in for the device
// array, not a device address: the device address is looked up once per
// device with cudaGetSymbolAddress, with that device current, during the first
// call made on it, and kept for the life of the process.  That first call may
// load this library's device module, so make it before any stream capture
// begins.  Do not use this entry point on a device after cudaDeviceReset: the
// module is reloaded and the kept address is no longer valid.
//
// Every call shares the one array and leaves the last call's contents in it.
// The arrival counters are cleared on the caller's stream before each launch;
// the partial tiles need no clearing (each split writes its whole tile before
// any split reads it).  Calls whose kernels overlap on the GPU (other streams,
// other host threads) race on the array and give wrong results: serialise them.
//
// A stream of an SM partition (goldy_partition_query) runs the GEMM inside
// the partition, as goldy_run does.
//
// Nothing here calls cudaMalloc, cudaFree or any allocating library routine.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <string>

#include "goldy_internal.h"

namespace goldy {

constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

goldy_status launch_planned_gemm(const GemmPlan& gp, const void* A, const void* B, void* C, unsigned char* ws,
                                 void* stream, size_t clear_off, size_t clear_bytes);

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
unsigned char* g_noalloc_addr[kMaxDevices] = {};

bool is_aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Device address of the scratch array on the current device (set up once).
goldy_status noalloc_scratch(unsigned char** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GOLDY_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(GOLDY_ERR_UNSUPPORTED, "device index too large");
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p)
      return fail(GOLDY_ERR_CUDA, std::string("cudaGetSymbolAddress(g_noalloc_scratch): ") + cudaGetErrorString(e));
    g_noalloc_addr[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_noalloc_addr[dev];
  return GOLDY_OK;
}
}  // namespace
}  // namespace goldy

using namespace goldy;

extern "C" goldy_status goldy_gemm_noalloc(const goldy_gemm_desc* desc, int variant, const void* A, const void* B,
                                           void* C, void* stream) {
  if (!desc) return fail(GOLDY_ERR_INVALID_ARG, "null descriptor");
  goldy_status st = check_desc(*desc, 0);
  if (st != GOLDY_OK) return st;
  if (variant < 0 || variant >= kNumVariants) return fail(GOLDY_ERR_INVALID_ARG, "variant id out of range");
  if (desc->batch != 1) return fail(GOLDY_ERR_UNSUPPORTED, "batched GEMMs go through goldy_run");

  GemmPlan gp;
  gp.desc = *desc;
  gp.variant = variant;
  const Variant v = variant_of(variant);
  const KindInfo& k = kKinds[v.kind];
  gp.kind = v.kind;
  gp.tiles_m = ceil_div(desc->M, tile_rows(k));
  gp.tiles_n = ceil_div(desc->N, tile_cols(k));
  gp.k_blocks = ceil_div(desc->K, kBlockK);
  gp.split = int(std::max<int64_t>(1, std::min<int64_t>(v.split, gp.k_blocks)));
  const int64_t tiles = gp.tiles_m * gp.tiles_n;
  gp.units = desc->K > 0 ? tiles * gp.split : 0;
  size_t need = 0, cnt_off = 0, counters = 0;
  if (gp.split > 1 && tiles > 0) {
    const size_t halves = k.pair ? 2 : 1;     // a CTA pair keeps a partial and a counter per CTA
    const size_t part = size_t(gp.units) * halves * kMmaM * k.mma_n * sizeof(float);
    cnt_off = (part + 255) & ~size_t(255);
    counters = size_t(tiles) * halves;
    need = cnt_off + counters * sizeof(uint32_t);
  }
  if (need > kNoAllocScratchBytes)
    return fail(GOLDY_ERR_INVALID_ARG, "this GEMM and variant need " + std::to_string(need) +
                                           " bytes of split-K scratch; the static scratch holds " +
                                           std::to_string(kNoAllocScratchBytes) +
                                           " bytes (use goldy_run with a workspace, or a smaller split)");
  if (desc->M == 0 || desc->N == 0) return ok();
  const size_t es = desc->c_dtype == GOLDY_BF16 ? 2 : 4;
  if (!C || !is_aligned(C, es)) return fail(GOLDY_ERR_INVALID_ARG, "C null or misaligned");
  if (desc->K > 0 && (!A || !B || !is_aligned(A, 16) || !is_aligned(B, 16)))
    return fail(GOLDY_ERR_INVALID_ARG, "A and B must be 16-byte aligned device pointers");

  unsigned char* scratch = nullptr;
  st = noalloc_scratch(&scratch);
  if (st != GOLDY_OK) return st;
  size_t clear_bytes = 0;
  if (need > 0) {
    gp.ws_part_off = 0;
    gp.ws_cnt_off = cnt_off;
    gp.ws_bytes = need;
    clear_bytes = counters * sizeof(uint32_t);
  }
  st = launch_planned_gemm(gp, A, B, C, scratch, stream, cnt_off, clear_bytes);
  if (st != GOLDY_OK) return st;
  return ok();
}

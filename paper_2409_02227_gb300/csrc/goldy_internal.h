// Internal host-side types shared by the planner (planner.cpp), the launch
// manager (runtime.cu) and the kernel instantiations (kernels.cu).  No CUDA
// types here: the planner is plain C++ and runs on machines without a GPU.
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "../../include/goldy.h"

namespace goldy {

// ---------------------------------------------------------------------------
// GO-Kernel kinds.  A kind fixes everything that is a template parameter of
// the kernel: the tensor-core tile (128 x mma_n, or its transpose for skinny
// M), the shared-memory pipeline depth and the number of accumulators kept in
// tensor memory.  Together these set the CTA's footprint on an SM — the
// trade-off between tile size, occupancy and on-chip memory the paper tunes
// per GEMM and per concurrency degree (Sec. 3.1, Sec. 4.2).
//   *_F ("full")  one CTA per SM, deepest pipeline
//   *_H ("half")  at most half of an SM's shared memory and tensor memory, so
//                 two CTAs (of this or of a co-running GEMM) fit on one SM
// ---------------------------------------------------------------------------
struct KindInfo {
  const char* name;
  int mma_n;       // tensor-core N (columns of the accumulator)
  int swap_ab;     // 1: tile is C^T (rows = 128 columns of C, cols = mma_n rows of C)
  int stages;      // shared-memory pipeline stages
  int acc_stages;  // accumulators in tensor memory (double buffering across tiles)
  int ctas_per_sm; // footprint target
  int pair;        // 1: a cluster of two CTAs computes 256-row tiles with one MMA (cta_group::2)
};

constexpr int kNumKinds = 11;
constexpr int kMmaM = 128;          // rows of every tensor-core tile
constexpr int kBlockK = 64;         // K elements per pipeline stage (one 128-byte row of bf16)
constexpr int kSplits[4] = {1, 2, 4, 8};
constexpr int kRcDivs[3] = {1, 2, 4};   // GPU, GPU/2, GPU/4 (Sec. 4.2.1)
constexpr int kNumVariants = kNumKinds * 4 * 3;
constexpr int kThreads = 192;       // 1 TMA warp, 1 MMA warp, 4 epilogue warps

inline constexpr KindInfo kKinds[kNumKinds] = {
    // name        mma_n swap stages acc ctas/SM pair
    {"n64_full", 64, 0, 8, 2, 1, 0},
    {"n64_half", 64, 0, 4, 2, 2, 0},
    {"n128_full", 128, 0, 5, 2, 1, 0},
    {"n128_half", 128, 0, 3, 2, 2, 0},
    {"n256_full", 256, 0, 4, 2, 1, 0},
    {"n256_half", 256, 0, 2, 1, 2, 0},
    {"t32_full", 32, 1, 8, 2, 1, 0},
    {"t32_half", 32, 1, 4, 2, 2, 0},
    {"t64_full", 64, 1, 8, 2, 1, 0},
    {"t64_half", 64, 1, 4, 2, 2, 0},
    {"p256_pair", 256, 0, 6, 2, 1, 1},   // 256 x 256 tiles over a CTA pair; split-K through the workspace
};

constexpr int stage_bytes(const KindInfo& k) {
  // a CTA of a pair holds 128 rows of A and half of the tile's B columns
  return kMmaM * kBlockK * 2 + (k.pair ? k.mma_n / 2 : k.mma_n) * kBlockK * 2;
}
constexpr int tmem_cols(const KindInfo& k) {
  int c = k.mma_n * k.acc_stages;
  int p = 32;
  while (p < c) p <<= 1;
  return p;
}
// Kinds with a whole SM to themselves (and the pair kind) store C through
// shared memory with TMA; they keep two 16 KB staging buffers.
constexpr bool epi_tma(const KindInfo& k) { return k.pair || (!k.swap_ab && k.ctas_per_sm == 1); }
// Kinds with a whole SM to themselves and tiles at most 128 wide reduce
// cluster split-K by pushing partial rows into receive slots of their peers:
// up to 7/8 of a 128 x mma_n fp32 tile (split 8).  The slots share one region
// with the TMA-store staging buffers (a launch uses one or the other).
constexpr int push_recv_bytes(const KindInfo& k) {
  return (!k.pair && k.ctas_per_sm == 1 && k.mma_n <= 128) ? 7 * kMmaM * k.mma_n * 4 / 8 : 0;
}
constexpr int epilogue_bytes(const KindInfo& k) {
  return (epi_tma(k) ? 2 * 16384 : 0) > push_recv_bytes(k) ? (epi_tma(k) ? 2 * 16384 : 0) : push_recv_bytes(k);
}
// stages, epilogue region, 1 KB for 1024-byte alignment of the swizzled
// tiles, 1 KB for barriers
constexpr int smem_bytes(const KindInfo& k) {
  return k.stages * stage_bytes(k) + epilogue_bytes(k) + 2048;
}

struct Variant {
  int id, kind, split, rc_div;
};
inline Variant variant_of(int id) {
  Variant v;
  v.id = id;
  v.kind = id / 12;
  v.split = kSplits[(id / 3) % 4];
  v.rc_div = kRcDivs[id % 3];
  return v;
}
inline int variant_id(int kind, int split_idx, int rc_idx) { return (kind * 4 + split_idx) * 3 + rc_idx; }

// Tile grid of one GEMM under a kind: the output is cut into tiles of
// (tile_m x tile_n) elements of C.
inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline int tile_rows(const KindInfo& k) { return k.pair ? 2 * kMmaM : (k.swap_ab ? k.mma_n : kMmaM); }
inline int tile_cols(const KindInfo& k) { return k.swap_ab ? kMmaM : k.mma_n; }
// rows of A one CTA loads per K block (the TMA box height)
inline int a_box_rows(const KindInfo& k) { return k.pair ? kMmaM : tile_rows(k); }

// ---------------------------------------------------------------------------
// Schedule
// ---------------------------------------------------------------------------
struct GemmPlan {
  goldy_gemm_desc desc;
  int group = 0;
  int variant = 0;
  int slot = 0;
  // derived at plan time (host integer work)
  int kind = 0;
  int split = 1;            // effective split: min(variant split, K blocks)
  int64_t tiles_m = 0, tiles_n = 0, k_blocks = 0;
  int64_t units = 0;        // tiles * split
  size_t ws_part_off = 0;   // byte offsets into the caller's workspace
  size_t ws_cnt_off = 0;
  size_t ws_bytes = 0;
  // a fused launch led by this GEMM may hand out its units through a pair of
  // counters here (fused schedules of several GEMMs; kNoOffset otherwise)
  size_t ws_dyn_off = ~size_t(0);
};

struct Group {
  int cd = 1;
  std::vector<int> members;  // launch order
};

struct Runtime;              // CUDA-side state (events), defined in runtime.cu

// Host stubs of the GO-Kernel of each kind, for fp32 (0) or bf16 (1) output,
// one GEMM per launch (fused = 0) or up to kMaxFused (fused = 1); kernels.cu
// is compiled once per kind (-DGOLDY_KIND=k) to define them.
constexpr int kMaxFused = 16;
const void* kernel_fn_k0(int out_bf16, int fused);
const void* kernel_fn_k1(int out_bf16, int fused);
const void* kernel_fn_k2(int out_bf16, int fused);
const void* kernel_fn_k3(int out_bf16, int fused);
const void* kernel_fn_k4(int out_bf16, int fused);
const void* kernel_fn_k5(int out_bf16, int fused);
const void* kernel_fn_k6(int out_bf16, int fused);
const void* kernel_fn_k7(int out_bf16, int fused);
const void* kernel_fn_k8(int out_bf16, int fused);
const void* kernel_fn_k9(int out_bf16, int fused);
const void* kernel_fn_k10(int out_bf16, int fused);

// Element-wise add (ewise.cu): Z = X + Y over n elements.
struct EwiseParams {
  const void* x;
  const void* y;
  void* z;
  int64_t n;
  int32_t vec_ok;   // all three pointers 16-byte aligned
  int32_t pad;
};
constexpr int kEwiseThreads = 256;
constexpr int kEwiseCtasPerSm = 8;
const void* ewise_kernel_fn(int bf16);

}  // namespace goldy

struct goldy_schedule {
  int flags = 0;
  int max_streams = 1;
  size_t workspace_bytes = 0;
  std::vector<goldy::GemmPlan> gemms;
  std::vector<goldy::Group> groups;
  goldy::Runtime* rt = nullptr;   // created on first goldy_run
};

// A GEMM co-scheduled with an element-wise add (planner.cpp builds it,
// runtime.cu runs it).
struct goldy_corun {
  goldy_schedule* gemm = nullptr;   // one GEMM with the chosen variant (owned)
  goldy_ewise_desc ew{};
  int policy = 0;
  int concurrent = 0;
  int add_rc_div = 1;
  goldy::Runtime* rt = nullptr;     // fork/join events, created on first run
};

namespace goldy {
// error text helpers (planner.cpp)
goldy_status fail(goldy_status st, const std::string& msg);
goldy_status ok();
// validation of one descriptor (planner.cpp)
goldy_status check_desc(const goldy_gemm_desc& d, int index);
// fill derived fields and workspace offsets (planner.cpp)
void finalize_schedule(goldy_schedule* s);
// release CUDA-side state (runtime.cu; no-op without it)
void runtime_release(Runtime* rt);
}  // namespace goldy

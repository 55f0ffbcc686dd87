// GO-Kernel: persistent, warp-specialised BF16 GEMM for sm_103a.
//
// What it computes (Sec. 2.1.2): C = A * B for A (M x K, row-major), B
// (K x N, row-major), fp32 accumulation, fp32 or bf16 (round-to-nearest-even)
// output; a strided-batched GEMM (Sec. 6.7's B-GEMMs) is `batch` such
// products at fixed strides, its tiles numbered batch entry by batch entry.
// Several GEMMs may share one launch (the launch's "units" are the
// concatenation of their tiles).
//
// How (Sec. 2.1.3's tiled GEMM re-expressed for tcgen05):
//   * The output is cut into tiles; a tile with its K-range split is a
//     "unit".  CTA b processes units b, b + gridDim.x, ... (persistent CTAs,
//     a static round-robin that is a function of the variant only).  The
//     grid size is the variant's resource constraint: capping it is how a
//     GO-Kernel leaves SMs to co-running GEMMs (Sec. 4.2.1).
//   * warp 0 (one thread): TMA producer.  Per 64-wide K block it loads the
//     A tile (K-major, 128-byte swizzle) and the B tile (N-major, 128-byte
//     swizzle) into a shared-memory ring of STAGES slots (mbarrier full/empty).
//   * warp 1 (one thread): allocates tensor memory, issues tcgen05.mma
//     (M = 128, N = MMA_N, K = 16 per instruction) into an fp32 accumulator
//     in tensor memory, ACC accumulators deep so the epilogue of one tile
//     overlaps the main loop of the next.
//   * warps 2-5: epilogue.  tcgen05.ld the accumulator (each warp its lane
//     quarter), convert and store to C.  With split-K, each split writes its
//     fp32 partial tile to the workspace; the last split to arrive (atomic
//     counter, no waiting on other CTAs) adds the partials in split order
//     0, 1, ..., S-1 and writes C, so every output element is summed in an
//     order fixed by the variant alone: results are bit-identical whether
//     the GEMM runs alone or next to others.
//   * SWAP (skinny M): the tensor-core tile is C^T — the 128-row MMA operand
//     is a slice of B's columns and the MMA_N-wide operand a slice of A's
//     rows — so an M of 16..64 still fills the 128-row tensor-core shape.
//
// Every wait is bounded (sm103_ptx.cuh).  A role that gives up raises the
// CTA's abort flag and the device error word, waits (bounded) for its own
// copies or MMAs in flight, and the CTA frees its tensor memory and exits.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cstdint>

#include "sm103_ptx.cuh"

namespace goldy {

struct GemmWork {
  void* c;              // output, row-major, ldc elements per row
  float* ws_part;       // split-K partial tiles (null when split == 1)
  uint32_t* ws_cnt;     // split-K arrival counter per tile
  int64_t ldc;
  int64_t c_bstride;    // elements between the C matrices of consecutive batch entries
  int32_t m, n, k;
  int32_t tiles_m, tiles_n;   // tiles of one batch entry
  int32_t split;        // K-range split, 1 <= split <= k_blocks
  int32_t k_blocks;     // ceil(K / 64)
  int32_t unit_begin;   // first unit of this GEMM within the launch
  int32_t c_tma;        // 1: C is written through tmap_c by TMA stores
  int32_t batch;        // strided batch entries (1: a plain GEMM)
};

// Where one batch entry's C lives: the store helpers' view of a GemmWork.
struct CView {
  void* c;
  int64_t ldc;
  int32_t m, n;
};

template <bool OUT_BF16>
__device__ __forceinline__ CView c_view(const GemmWork& w, int b) {
  CView v;
  v.c = static_cast<char*>(w.c) + int64_t(b) * w.c_bstride * (OUT_BF16 ? 2 : 4);
  v.ldc = w.ldc;
  v.m = w.m;
  v.n = w.n;
  return v;
}

template <int MAXG>
struct LaunchParams {
  CUtensorMap tmap_a[MAXG];   // A: dims {K, M, batch}, box {64, rows of the A tile, 1}
  CUtensorMap tmap_b[MAXG];   // B: dims {N, K, batch}, box {64, 64, 1}
  CUtensorMap tmap_c[MAXG];   // C: dims {N, M, batch}, box {128-byte row, 128 rows, 1} (when g[].c_tma)
  GemmWork g[MAXG];
  int32_t n_gemms;
  int32_t total_units;
  int* err;                   // device error word (first failure wins)
  unsigned long long* trace;  // optional phase trace, kTracePerCta stamps per CTA (null: off)
  int32_t cluster;            // 0, or the split-K factor S of every GEMM in the launch when the
                              // launch is made of clusters of S CTAs (the splits of one tile)
  uint32_t* dyn;              // null: CTA b takes units b, b + grid, ...; else a zeroed pair of
                              // counters (units taken, CTAs done): after its first unit b a CTA
                              // takes grid + (counter++), and the last CTA to leave zeroes both
  uint64_t wait_ns;           // limit of every bounded wait (0: ptx::kWaitLimitNs)
  int32_t early_loads;        // 1: the load and MMA roles start before the previous kernel on the
                              // stream has completed (the caller asserted that no earlier kernel
                              // writes this launch's A or B); C and the workspace are still
                              // touched only after it (griddepcontrol.wait in the epilogue)
  int32_t stall_test;         // test hook: CTA 0's producer never fills its first stage, so the
                              // MMA thread's bounded wait for it runs out (0 in normal use)
};

// Units a CTA has taken but its MMA thread and epilogue have not yet both
// read, at most (a ring of unit indices in shared memory, used when the
// launch hands units out from a counter; with the static round-robin every
// role computes the sequence itself).
constexpr int kUnitRing = 8;

// Phase trace (optional, for profiling): %globaltimer stamps per CTA.
enum : int {
  kTrStart = 0,        // kernel entry
  kTrSetup = 1,        // the epilogue is past the wait for the previous grid (set-up done)
  kTrFirstLoad = 2,    // producer issued its first TMA load
  kTrFirstFull = 3,    // MMA thread saw its first full stage
  kTrFirstMmaDone = 4, // MMA thread committed its first accumulator
  kTrFirstAcc = 5,     // epilogue saw its first accumulator
  kTrPartials = 6,     // split-K: partial tile stored and fenced
  kTrArrived = 7,      // split-K: arrival counter bumped
  kTrFirstStore = 8,   // epilogue finished its first unit
  kTrEnd = 9,          // all roles done
  kTrPreWait = 10,     // set-up done, about to wait for the grid this launch depends on
  kTrProducerGo = 11,  // producer starts its first unit
  kTrGrid = 12,        // grid size of the launch (launches of one run trace into consecutive regions)
  kTrCta = 13,         // CTA index within its launch
  kTrUnits = 14,       // units processed by this CTA
  kTrSm = 15,          // SM id
  kTracePerCta = 16,
};

enum : int {
  kErrProducerWait = 1,
  kErrMmaWait = 2,
  kErrEpilogueWait = 3,
  kErrClusterWait = 4,
};

struct UnitCoord {
  int g, tile, s, b, tm, tn, kb0, kb1;   // tile counts over all batch entries; b = batch entry
};

template <int MAXG>
__device__ __forceinline__ UnitCoord decode_unit(const LaunchParams<MAXG>& p, int u) {
  UnitCoord c;
  int g = 0;
#pragma unroll 1
  while (g + 1 < p.n_gemms && u >= p.g[g + 1].unit_begin) ++g;
  const GemmWork& w = p.g[g];
  const int local = u - w.unit_begin;
  c.g = g;
  c.tile = local / w.split;
  c.s = local - c.tile * w.split;
  const int per_batch = w.tiles_m * w.tiles_n;
  c.b = c.tile / per_batch;
  const int t = c.tile - c.b * per_batch;
  c.tm = t % w.tiles_m;
  c.tn = t / w.tiles_m;
  c.kb0 = (c.s * w.k_blocks) / w.split;
  c.kb1 = ((c.s + 1) * w.k_blocks) / w.split;
  return c;
}

// The fields of a GemmWork that decode a unit, copied into shared memory at
// set-up: the kernel parameter block is several kilobytes (tensor maps
// first), and reading these fields from it on the producer's critical path
// measured ~0.4 us before the first load of a launch.
struct UnitTable {
  int32_t unit_begin, split, tiles_m, tiles_n, k_blocks;
};

__device__ __forceinline__ UnitCoord decode_unit_tab(const UnitTable* t, int n_gemms, int u) {
  UnitCoord c;
  int g = 0;
#pragma unroll 1
  while (g + 1 < n_gemms && u >= t[g + 1].unit_begin) ++g;
  const UnitTable& w = t[g];
  const int local = u - w.unit_begin;
  c.g = g;
  c.tile = local / w.split;
  c.s = local - c.tile * w.split;
  const int per_batch = w.tiles_m * w.tiles_n;
  c.b = c.tile / per_batch;
  const int t2 = c.tile - c.b * per_batch;
  c.tm = t2 % w.tiles_m;
  c.tn = t2 / w.tiles_m;
  c.kb0 = (c.s * w.k_blocks) / w.split;
  c.kb1 = ((c.s + 1) * w.k_blocks) / w.split;
  return c;
}

__device__ __forceinline__ void trace_stamp(unsigned long long* trace, int slot) {
  if (trace) trace[blockIdx.x * kTracePerCta + slot] = ptx::global_timer();
}

__device__ __forceinline__ void raise_error(int* err, volatile int* abort_flag, int code) {
  *abort_flag = 1;
  if (err) atomicCAS(err, 0, code);
}

// Store 32 consecutive accumulator columns of one accumulator row.
//  !SWAP: row `r` of the tile is C row m0 + r; columns n0 + c0 .. +31.
//   SWAP: row `r` of the tile is C column n0 + r; columns are C rows m0 + c0 .. +31.
template <bool SWAP, bool OUT_BF16>
__device__ __forceinline__ void store_chunk(const CView& w, int m0, int n0, int r, int c0, const float (&v)[32]) {
  if (!SWAP) {
    const int64_t row = int64_t(m0) + r;
    if (row >= w.m) return;
    const int col0 = n0 + c0;
    if (OUT_BF16) {
      __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(w.c) + row * w.ldc + col0;
      if (col0 + 32 <= w.n && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 pk;
          __nv_bfloat162 h0 = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
          __nv_bfloat162 h1 = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
          __nv_bfloat162 h2 = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
          __nv_bfloat162 h3 = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
          pk.x = *reinterpret_cast<uint32_t*>(&h0);
          pk.y = *reinterpret_cast<uint32_t*>(&h1);
          pk.z = *reinterpret_cast<uint32_t*>(&h2);
          pk.w = *reinterpret_cast<uint32_t*>(&h3);
          reinterpret_cast<uint4*>(dst)[q] = pk;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (col0 + j < w.n) dst[j] = __float2bfloat16_rn(v[j]);
      }
    } else {
      float* dst = static_cast<float*>(w.c) + row * w.ldc + col0;
      if (col0 + 32 <= w.n && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          reinterpret_cast<float4*>(dst)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (col0 + j < w.n) dst[j] = v[j];
      }
    }
  } else {
    const int64_t col = int64_t(n0) + r;
    if (col >= w.n) return;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int64_t row = int64_t(m0) + c0 + j;
      if (row < w.m) {
        if (OUT_BF16)
          static_cast<__nv_bfloat16*>(w.c)[row * w.ldc + col] = __float2bfloat16_rn(v[j]);
        else
          static_cast<float*>(w.c)[row * w.ldc + col] = v[j];
      }
    }
  }
}

// Store 4 consecutive accumulator columns (acc_col .. acc_col+3) of
// accumulator row acc_row, mapped to C as in store_chunk.
template <bool SWAP, bool OUT_BF16>
__device__ __forceinline__ void store_quad(const CView& w, int m0, int n0, int acc_row, int acc_col, float4 a) {
  const float v[4] = {a.x, a.y, a.z, a.w};
  if (!SWAP) {
    const int64_t row = int64_t(m0) + acc_row;
    if (row >= w.m) return;
    const int col0 = n0 + acc_col;
    if (OUT_BF16) {
      __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(w.c) + row * w.ldc + col0;
      if (col0 + 4 <= w.n && (reinterpret_cast<uintptr_t>(dst) & 7) == 0) {
        __nv_bfloat162 h0 = __floats2bfloat162_rn(v[0], v[1]);
        __nv_bfloat162 h1 = __floats2bfloat162_rn(v[2], v[3]);
        uint2 pk;
        pk.x = *reinterpret_cast<uint32_t*>(&h0);
        pk.y = *reinterpret_cast<uint32_t*>(&h1);
        *reinterpret_cast<uint2*>(dst) = pk;
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (col0 + j < w.n) dst[j] = __float2bfloat16_rn(v[j]);
      }
    } else {
      float* dst = static_cast<float*>(w.c) + row * w.ldc + col0;
      if (col0 + 4 <= w.n && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
        *reinterpret_cast<float4*>(dst) = a;
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (col0 + j < w.n) dst[j] = v[j];
      }
    }
  } else {
    const int64_t col = int64_t(n0) + acc_row;
    if (col >= w.n) return;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t row = int64_t(m0) + acc_col + j;
      if (row < w.m) {
        if (OUT_BF16)
          static_cast<__nv_bfloat16*>(w.c)[row * w.ldc + col] = __float2bfloat16_rn(v[j]);
        else
          static_cast<float*>(w.c)[row * w.ldc + col] = v[j];
      }
    }
  }
}

// Cluster split-K: this CTA (split `rank` of S) sums rows rank*128/S ..
// (rank+1)*128/S - 1 of the tile over all S partial tiles, in split order
// 0, 1, ..., S-1, and stores them.  Partial layout: [chunk][float4][row].
// Per batch, IB items x S partials are loaded before any is added.
template <int MMA_N, int S, bool SWAP, bool OUT_BF16>
__device__ __forceinline__ void reduce_slice(const CView& w, const float4* tile_parts, int rank, int m0, int n0,
                                             int t) {
  constexpr int R = 128 / S;
  constexpr int COLS4 = MMA_N / 4;
  constexpr int PER_THREAD = R * COLS4 / 128;
  constexpr int IB = (16 / S < PER_THREAD) ? 16 / S : PER_THREAD;
  constexpr int TILE_F4 = 128 * MMA_N / 4;
  static_assert(PER_THREAD >= 1 && PER_THREAD % IB == 0, "reduce tiling");
  const int r0 = rank * R;
#pragma unroll 1
  for (int k0 = 0; k0 < PER_THREAD; k0 += IB) {
    float4 vals[IB][S];
#pragma unroll
    for (int b = 0; b < IB; ++b) {
      const int i = t + 128 * (k0 + b);
      const int off = (i / R) * 128 + r0 + (i % R);
#pragma unroll
      for (int s2 = 0; s2 < S; ++s2) vals[b][s2] = __ldcg(&tile_parts[size_t(s2) * TILE_F4 + off]);
    }
#pragma unroll
    for (int b = 0; b < IB; ++b) {
      const int i = t + 128 * (k0 + b);
      float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int s2 = 0; s2 < S; ++s2) {
        a.x += vals[b][s2].x;
        a.y += vals[b][s2].y;
        a.z += vals[b][s2].z;
        a.w += vals[b][s2].w;
      }
      store_quad<SWAP, OUT_BF16>(w, m0, n0, r0 + (i % R), 4 * (i / R), a);
    }
  }
}

// Store one accumulator tile (128 rows x MMA_N columns, rows m0.., columns
// n0..) through shared memory with TMA.  Per chunk of 128-byte rows (32 fp32
// or 64 bf16 columns) every thread writes its row into a staging buffer with
// the 128-byte swizzle (so a warp's writes hit distinct banks), then one
// thread issues the tensor store; two 16 KB buffers alternate, and a buffer
// is reused only after the store two chunks back has read it.  WIDE: the
// chunks go to consecutive 16 KB buffers from `staging` on (MMA_N * 512 bytes
// for fp32, half that for bf16), none reused, and only the staging is done
// here (shared memory only; issue_tile_wide stores them) — for a CTA's last
// tile, staged in its idle operand ring.  The store clips rows and columns
// outside C.
template <int MMA_N, bool OUT_BF16, bool WIDE = false>
__device__ __forceinline__ void store_tile_tma(const void* tmap_c, uint32_t staging, uint32_t& stg, uint32_t taddr,
                                               int r, int et, int m0, int n0, int b) {
  constexpr int CHUNK = OUT_BF16 ? 64 : 32;
#pragma unroll 1
  for (int c0 = 0; c0 < MMA_N; c0 += CHUNK) {
    const uint32_t buf = WIDE ? staging + uint32_t(c0 / CHUNK) * 16384u : staging + (stg & 1u) * 16384u;
    if (!WIDE && et == 0) ptx::bulk_wait_group_read<1>();
    ptx::named_bar_sync(1, 128);
    const uint32_t row = buf + uint32_t(r) * 128u;
    const uint32_t sw = uint32_t(r & 7);
    uint32_t raw[32];
    __syncwarp();
    ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
    ptx::tmem_ld_wait();
    if (!OUT_BF16) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        ptx::st_shared_v4(row + ((uint32_t(j) ^ sw) << 4), raw[4 * j], raw[4 * j + 1], raw[4 * j + 2], raw[4 * j + 3]);
    } else {
      uint32_t pk[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(raw[2 * j]), __uint_as_float(raw[2 * j + 1]));
        pk[j] = *reinterpret_cast<uint32_t*>(&h);
      }
      __syncwarp();
      ptx::tmem_ld_32x32b_x32(taddr + c0 + 32, raw);
      ptx::tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 4; ++j)
        ptx::st_shared_v4(row + ((uint32_t(j) ^ sw) << 4), pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(raw[2 * j]), __uint_as_float(raw[2 * j + 1]));
        pk[j] = *reinterpret_cast<uint32_t*>(&h);
      }
#pragma unroll
      for (int j = 0; j < 4; ++j)
        ptx::st_shared_v4(row + ((uint32_t(j + 4) ^ sw) << 4), pk[4 * j], pk[4 * j + 1], pk[4 * j + 2],
                          pk[4 * j + 3]);
    }
    ptx::fence_proxy_async_smem();
    if (WIDE) continue;
    ptx::named_bar_sync(1, 128);
    if (et == 0) {
      ptx::tma_store_3d(tmap_c, buf, n0 + c0, m0, b);
      ptx::bulk_commit_group();
    }
    ++stg;
  }
  if (WIDE) ptx::named_bar_sync(1, 128);   // every chunk staged and fenced
}

// The tensor stores of a tile staged by store_tile_tma<..., true> (one
// thread issues them all, one bulk group).
template <int MMA_N, bool OUT_BF16>
__device__ __forceinline__ void issue_tile_wide(const void* tmap_c, uint32_t staging, int et, int m0, int n0, int b) {
  constexpr int CHUNK = OUT_BF16 ? 64 : 32;
  if (et != 0) return;
#pragma unroll 1
  for (int c0 = 0; c0 < MMA_N; c0 += CHUNK)
    ptx::tma_store_3d(tmap_c, staging + uint32_t(c0 / CHUNK) * 16384u, n0 + c0, m0, b);
  ptx::bulk_commit_group();
}

// Shared-memory layout of a whole fp32 partial tile for the on-chip cluster
// reduction: row-major, MMA_N / 4 granules of 16 bytes per row, granule f of
// row r stored at position f ^ (r & 7) — a thread writing its accumulator row
// and a warp reading consecutive granules of one row both hit distinct banks.
template <int MMA_N>
__device__ __forceinline__ uint32_t part_offset(int r, int f) {
  return uint32_t(r * (MMA_N / 4) + (f ^ (r & 7))) * 16u;
}

// Cluster split-K with the partial tiles in shared memory: this CTA (split
// `rank` of S) sums rows rank*128/S .. (rank+1)*128/S - 1 of the tile over
// the S partials, partial s read from the shared memory of cluster CTA s, in
// split order 0, 1, ..., S-1.  Consecutive threads take consecutive 16-byte
// granules of a row, so C is written in whole rows.
template <int MMA_N, int S, bool SWAP, bool OUT_BF16>
__device__ __forceinline__ void reduce_slice_dsmem(const CView& w, uint32_t part_smem, int rank, int m0, int n0,
                                                   int t) {
  constexpr int R = 128 / S;
  constexpr int G4 = MMA_N / 4;                 // granules per row
  constexpr int PER_THREAD = R * G4 / 128;
  constexpr int IB = (16 / S < PER_THREAD) ? 16 / S : PER_THREAD;
  static_assert(PER_THREAD >= 1 && PER_THREAD % IB == 0, "reduce tiling");
  const int r0 = rank * R;
  uint32_t peer[S];
#pragma unroll
  for (int s2 = 0; s2 < S; ++s2) peer[s2] = ptx::map_to_rank(part_smem, uint32_t(s2));
#pragma unroll 1
  for (int k0 = 0; k0 < PER_THREAD; k0 += IB) {
    float4 vals[IB][S];
#pragma unroll
    for (int b = 0; b < IB; ++b) {
      const int i = t + 128 * (k0 + b);
      const uint32_t off = part_offset<MMA_N>(r0 + i / G4, i % G4);
#pragma unroll
      for (int s2 = 0; s2 < S; ++s2) vals[b][s2] = ptx::ld_shared_cluster_v4(peer[s2] + off);
    }
#pragma unroll
    for (int b = 0; b < IB; ++b) {
      const int i = t + 128 * (k0 + b);
      float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int s2 = 0; s2 < S; ++s2) {
        a.x += vals[b][s2].x;
        a.y += vals[b][s2].y;
        a.z += vals[b][s2].z;
        a.w += vals[b][s2].w;
      }
      store_quad<SWAP, OUT_BF16>(w, m0, n0, r0 + i / G4, 4 * (i % G4), a);
    }
  }
}

// Layout of a slice (R rows x MMA_N fp32 columns) of the pushed reduction:
// column-chunk major, so that each 32-column chunk of a slice is one
// contiguous R x 128-byte block that can be sent as soon as it is staged;
// within a chunk, granule j of row rr sits at j ^ (rr & 7) (a thread writing
// its row and a warp reading consecutive granules both spread over the banks).
__device__ __forceinline__ uint32_t push_offset(int rr, int f, int R) {
  return uint32_t((f >> 3) * R * 128 + rr * 128 + (((f & 7) ^ (rr & 7)) << 4));
}

// Cluster split-K with pushed partials: CTA s of the S splits of a tile owns
// rows s*128/S .. (s+1)*128/S - 1.  Every CTA sends the rows it does not own
// to their owner (a bulk copy into the owner's receive slot, counted on the
// owner's mbarrier) and keeps its own rows in its ring; the owner then sums,
// from its own shared memory, the S partials of its rows in split order
// 0, 1, ..., S-1 and stores them.  A slot holds 128/S rows in the layout of
// push_offset; sender s goes to slot s (s < owner) or s - 1 (s > owner).
template <int MMA_N, int S, bool SWAP, bool OUT_BF16>
__device__ __forceinline__ void reduce_slice_pushed(const CView& w, uint32_t own_slot, uint32_t recv_slots, int rank,
                                                    int m0, int n0, int t) {
  constexpr int R = 128 / S;
  constexpr int G4 = MMA_N / 4;
  constexpr int PER_THREAD = R * G4 / 128;
  constexpr uint32_t SLOT_BYTES = uint32_t(R * MMA_N * 4);
  static_assert(PER_THREAD >= 1 && (R * G4) % 128 == 0, "reduce tiling");
  uint32_t src[S];
#pragma unroll
  for (int s2 = 0; s2 < S; ++s2)
    src[s2] = s2 == rank ? own_slot : recv_slots + uint32_t(s2 < rank ? s2 : s2 - 1) * SLOT_BYTES;
#pragma unroll 2
  for (int k = 0; k < PER_THREAD; ++k) {
    const int i = t + 128 * k;
    const uint32_t off = push_offset(i / G4, i % G4, R);
    float4 v[S];
#pragma unroll
    for (int s2 = 0; s2 < S; ++s2) v[s2] = ptx::ld_shared_v4(src[s2] + off);
    float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
    for (int s2 = 0; s2 < S; ++s2) {
      a.x += v[s2].x;
      a.y += v[s2].y;
      a.z += v[s2].z;
      a.w += v[s2].w;
    }
    store_quad<SWAP, OUT_BF16>(w, m0, n0, rank * R + i / G4, 4 * (i % G4), a);
  }
}

// Bytes of the receive slots of the pushed reduction: the largest split
// (8) leaves 7/8 of a 128 x MMA_N fp32 tile to receive.  Kinds that own a
// whole SM with MMA_N <= 128 have room for them (the host's shared-memory
// size per kind reserves the same bytes).
template <int MMA_N, int MIN_CTAS>
struct PushRecv {
  static constexpr bool enabled = MIN_CTAS == 1 && MMA_N <= 128;
  static constexpr int bytes = enabled ? 7 * 128 * MMA_N * 4 / 8 : 0;
};

template <int MMA_N, int ACC>
struct TmemCols {
  static constexpr uint32_t need = uint32_t(MMA_N * ACC);
  static constexpr uint32_t value = need <= 32 ? 32 : need <= 64 ? 64 : need <= 128 ? 128 : need <= 256 ? 256 : 512;
};

template <int MMA_N, bool SWAP, int STAGES, int ACC, bool OUT_BF16, int MAXG, int MIN_CTAS, bool EPI_TMA>
__global__ void __launch_bounds__(192, MIN_CTAS) go_gemm_kernel(const __grid_constant__ LaunchParams<MAXG> p) {
  constexpr int X_BYTES = 128 * 64 * 2;              // MMA operand A: 128 rows x 64 K
  constexpr int Y_BYTES = MMA_N * 64 * 2;            // MMA operand B: MMA_N rows x 64 K
  constexpr int STAGE_BYTES = X_BYTES + Y_BYTES;
  constexpr int TILE_M = SWAP ? MMA_N : 128;         // C rows per tile
  constexpr int TILE_N = SWAP ? 128 : MMA_N;         // C columns per tile
  constexpr int B_BOXES = TILE_N / 64;               // 64-column TMA boxes of B per stage
  // a CTA's last tile can be staged whole in the operand ring (see the epilogue)
  constexpr bool kWideFits = !SWAP && STAGES * STAGE_BYTES >= 128 * MMA_N * (OUT_BF16 ? 2 : 4);
  constexpr uint32_t TMEM_COLS = TmemCols<MMA_N, ACC>::value;
  // !SWAP: MMA-A = A tile (K-major), MMA-B = B tile (N-major)
  //  SWAP: MMA-A = B tile (N-major), MMA-B = A tile (K-major)
  constexpr uint32_t IDESC = ptx::make_idesc_bf16(128, MMA_N, SWAP ? 1 : 0, SWAP ? 0 : 1);
  constexpr uint32_t KMAJ_STEP = 32;                 // bytes per 16 K elements, K-major
  constexpr uint32_t MNMAJ_STEP = 2048;              // bytes per 16 K rows, N-major
  constexpr uint32_t MNMAJ_LBO = 64 * 128;           // bytes between 64-wide N chunks
  static_assert(MMA_N % 32 == 0 && MMA_N >= 32 && MMA_N <= 256, "MMA_N");
  static_assert(TILE_N % 64 == 0, "B tiles are whole 64-column boxes");
  static_assert(STAGES <= 32, "stage bitmasks");
  static_assert(!(EPI_TMA && SWAP), "the TMA-store epilogue writes untransposed tiles");
  constexpr int STAGING_BYTES = EPI_TMA ? 2 * 16384 : 0;
  // a whole fp32 partial tile fits in the ring's shared memory
  constexpr bool kPartFitsRing = STAGES * STAGE_BYTES >= 128 * MMA_N * 4;
  // pushed cluster reduction: receive slots share the region after the ring
  // with the TMA-store staging buffers (a launch uses one or the other: the
  // pushed reduction runs only when every GEMM of the launch is split)
  constexpr bool kPush = PushRecv<MMA_N, MIN_CTAS>::enabled;
  constexpr int EPI_BYTES =
      STAGING_BYTES > PushRecv<MMA_N, MIN_CTAS>::bytes ? STAGING_BYTES : PushRecv<MMA_N, MIN_CTAS>::bytes;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES + EPI_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* tfull = bars + 2 * STAGES;
  uint64_t* tempty = bars + 2 * STAGES + ACC;
  uint64_t* drain = bars + 2 * STAGES + 2 * ACC;
  uint64_t* redbar = drain + 1;        // cluster split-K: 2 barriers, alternating by unit
  uint64_t* recvbar = redbar + 2;      // pushed cluster reduction: bytes received
  uint64_t* ufull = recvbar + 1;       // unit ring: the producer published the unit index
  uint64_t* uempty = ufull + kUnitRing;  // unit ring: the MMA thread and the epilogue read it
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(uempty + kUnitRing);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);
  volatile int* units_taken = reinterpret_cast<volatile int*>(tmem_slot + 3);
  UnitTable* utab = reinterpret_cast<UnitTable*>(tmem_slot + 4);   // MAXG entries, inside the 1 KB barrier area
  volatile int* uring = reinterpret_cast<volatile int*>(utab + MAXG);   // kUnitRing unit indices
  static_assert((2 * STAGES + 2 * ACC + 4 + 2 * kUnitRing) * 8 + 16 + MAXG * int(sizeof(UnitTable)) +
                        kUnitRing * 4 <= 1024,
                "barrier area");
  const int n_gemms = p.n_gemms;

  const uint32_t tiles_base = ptx::smem_u32(smem);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  unsigned long long* const trace = p.trace;
  // the next launch on this stream may start its set-up now; it waits
  // (griddep_wait) for this grid to complete before touching global memory
  ptx::griddep_launch_dependents();

  // pushed cluster reduction: one unit per CTA, every GEMM split S = cluster
  const bool push_on = kPush && p.cluster > 0 && p.total_units == int(gridDim.x);

  if (threadIdx.x == 0) {
    trace_stamp(trace, kTrStart);
    // start fetching the TMA descriptors before anything else: the first
    // load waits on them
    for (int g = 0; g < p.n_gemms; ++g) {
      ptx::prefetch_tensormap(&p.tmap_a[g]);
      ptx::prefetch_tensormap(&p.tmap_b[g]);
    }
    if (trace) {
      uint32_t sm;
      asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
      trace[blockIdx.x * kTracePerCta + kTrSm] = sm;
      trace[blockIdx.x * kTracePerCta + kTrGrid] = gridDim.x;
      trace[blockIdx.x * kTracePerCta + kTrCta] = blockIdx.x;
    }
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(ptx::smem_u32(&full[s]), 1);
      ptx::mbar_init(ptx::smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < ACC; ++a) {
      ptx::mbar_init(ptx::smem_u32(&tfull[a]), 1);
      ptx::mbar_init(ptx::smem_u32(&tempty[a]), 128);
    }
    ptx::mbar_init(ptx::smem_u32(drain), 1);
    if (p.cluster > 0) {
      ptx::mbar_init(ptx::smem_u32(&redbar[0]), uint32_t(p.cluster));
      ptx::mbar_init(ptx::smem_u32(&redbar[1]), uint32_t(p.cluster));
    }
    if (push_on) ptx::mbar_init(ptx::smem_u32(recvbar), 1);
    for (int q = 0; q < kUnitRing; ++q) {
      ptx::mbar_init(ptx::smem_u32(&ufull[q]), 1);
      ptx::mbar_init(ptx::smem_u32(&uempty[q]), 2);
    }
    *abort_flag = 0;
    *last_flag = 0;
    *units_taken = 0;
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
    // the phase completes once the S - 1 peers' rows of this CTA's slice
    // have landed (peers start sending only after the cluster-wide sync below)
    if (push_on)
      ptx::mbar_arrive_expect_tx(ptx::smem_u32(recvbar),
                                 uint32_t((p.cluster - 1) * (128 / p.cluster) * MMA_N * 4));
  }
  if (warp == 1) {
    ptx::tmem_alloc(ptx::smem_u32(tmem_slot), TMEM_COLS);
    ptx::tmem_relinquish();
  } else if (warp == 2) {
    for (int g = lane; g < p.n_gemms; g += 32) {
      UnitTable e;
      e.unit_begin = p.g[g].unit_begin;
      e.split = p.g[g].split;
      e.tiles_m = p.g[g].tiles_m;
      e.tiles_n = p.g[g].tiles_n;
      e.k_blocks = p.g[g].k_blocks;
      utab[g] = e;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  // peers signal this CTA's reduction barriers: every CTA of the cluster must
  // have initialised them before any signal is sent
  if (p.cluster > 0) ptx::cluster_sync_all();
  const uint32_t tmem_base = *tmem_slot;
  const uint64_t wlim = p.wait_ns ? p.wait_ns : ptx::kWaitLimitNs;
  if (threadIdx.x == 0) trace_stamp(trace, kTrPreWait);
  // set-up above touched only shared and tensor memory; global memory (the
  // operands, C, the split-K workspace) only after the previous grid is done.
  // Early mode: the producer (reading A and B only, asserted not written by
  // an earlier kernel) and the MMA thread (shared and tensor memory only)
  // go ahead; the epilogue, which writes C and the workspace, still waits.
  // A launch that hands units out from a workspace counter loads its first
  // unit (this CTA's own) early too; the producer waits before its first
  // read of the counter, which the previous launch over the same GEMMs
  // zeroes as it ends.
  const bool early = p.early_loads != 0 && warp < 2;
  // In early mode the epilogue waits where it first writes global memory
  // (below): a CTA's last tile is read out of tensor memory into the idle
  // operand ring before that wait, so only its stores are left after it.
  const bool epi_defer = p.early_loads != 0 && warp >= 2;
  if (!early && !epi_defer) ptx::griddep_wait();
  if (threadIdx.x == 64 && !epi_defer) trace_stamp(trace, kTrSetup);   // the first epilogue thread waits

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ producer
      int stage = 0;
      uint32_t phase = 0, issued = 0, last_phase = 0;
      bool ok = true, stalled = false;
      int u = blockIdx.x, taken = 0;
      for (int seq = 0; ok && !stalled; ++seq) {
        if (p.dyn) {
          // publish the unit (or the end: an index past the last unit) to
          // the MMA thread and the epilogue
          const int slot = seq % kUnitRing;
          if (seq >= kUnitRing &&
              !ptx::mbar_wait(ptx::smem_u32(&uempty[slot]), uint32_t((seq / kUnitRing) - 1) & 1u, abort_flag,
                              wlim)) {
            ok = false;
            break;
          }
          uring[slot] = u;
          ptx::mbar_arrive(ptx::smem_u32(&ufull[slot]));
        }
        if (u >= p.total_units) break;
        ++taken;
        // the next unit, taken now so that the counter's latency overlaps
        // this unit's loads — except after an early start, where the counter
        // is read once the first unit's loads are out and the previous grid
        // is done
        const bool defer_next = p.dyn && early && seq == 0;
        int next = defer_next ? 0 : (p.dyn ? int(gridDim.x + atomicAdd(p.dyn, 1u)) : u + int(gridDim.x));
        if (issued == 0) trace_stamp(trace, kTrProducerGo);
        const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
        const void* ta = &p.tmap_a[c.g];
        const void* tb = &p.tmap_b[c.g];
        const int m0 = c.tm * TILE_M;
        const int n0 = c.tn * TILE_N;
        for (int kb = c.kb0; kb < c.kb1; ++kb) {
          // a slot is waited for only once it has been filled before: on the
          // first pass the ring is empty (waiting on a fresh barrier's
          // preceding phase measured ~0.7 us before the first load)
          if ((issued >> stage & 1) && !ptx::mbar_wait(ptx::smem_u32(&empty[stage]), phase ^ 1, abort_flag, wlim)) {
            ok = false;
            break;
          }
          if (p.stall_test && blockIdx.x == 0 && issued == 0) {
            // test hook: the first stage is never filled.  No copy is in
            // flight and no address is touched; the MMA thread's bounded
            // wait for the stage runs out and raises the abort flag, which
            // ends this wait too.
            const uint64_t t0 = ptx::global_timer();
            while (!*abort_flag && ptx::global_timer() - t0 < 4 * wlim) {
            }
            stalled = true;
            break;
          }
          const uint32_t fb = ptx::smem_u32(&full[stage]);
          ptx::mbar_arrive_expect_tx(fb, STAGE_BYTES);
          const uint32_t xs = tiles_base + stage * STAGE_BYTES;
          const uint32_t ys = xs + X_BYTES;
          const int k0 = kb * 64;
          if (!SWAP) {
            ptx::tma_load_3d(xs, ta, fb, k0, m0, c.b);
#pragma unroll
            for (int j = 0; j < B_BOXES; ++j) ptx::tma_load_3d(ys + j * 8192, tb, fb, n0 + 64 * j, k0, c.b);
          } else {
#pragma unroll
            for (int j = 0; j < B_BOXES; ++j) ptx::tma_load_3d(xs + j * 8192, tb, fb, n0 + 64 * j, k0, c.b);
            ptx::tma_load_3d(ys, ta, fb, k0, m0, c.b);
          }
          if (issued == 0) trace_stamp(trace, kTrFirstLoad);
          issued |= 1u << stage;
          last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (defer_next) {
          if (!ok || stalled) break;
          ptx::griddep_wait();
          next = int(gridDim.x + atomicAdd(p.dyn, 1u));
        }
        u = next;
      }
      *units_taken = taken;
      if (!ok) {
        raise_error(p.err, abort_flag, kErrProducerWait);
        // let every copy this thread started land before the CTA can exit
        for (int s = 0; s < STAGES; ++s)
          if (issued >> s & 1) ptx::mbar_wait(ptx::smem_u32(&full[s]), (last_phase >> s) & 1, nullptr);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------- MMA issuer
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0, acc_used = 0;
      bool ok = true, any = false;
      for (int seq = 0; ok; ++seq) {
        int u = int(blockIdx.x) + seq * int(gridDim.x);   // static round-robin
        if (p.dyn) {
          const int slot = seq % kUnitRing;
          if (!ptx::mbar_wait(ptx::smem_u32(&ufull[slot]), uint32_t(seq / kUnitRing) & 1u, abort_flag, wlim)) {
            ok = false;
            break;
          }
          u = uring[slot];
          ptx::mbar_arrive(ptx::smem_u32(&uempty[slot]));
        }
        if (u >= p.total_units) break;
        const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
        // an accumulator is waited for only once it has been used before
        if ((acc_used >> acc & 1) &&
            !ptx::mbar_wait(ptx::smem_u32(&tempty[acc]), acc_phase ^ 1, abort_flag, wlim)) {
          ok = false;
          break;
        }
        acc_used |= 1u << acc;
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + uint32_t(acc * MMA_N);
        for (int kb = c.kb0; kb < c.kb1; ++kb) {
          if (!ptx::mbar_wait(ptx::smem_u32(&full[stage]), phase, abort_flag, wlim)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          if (!any) trace_stamp(trace, kTrFirstFull);
          const uint32_t xs = tiles_base + stage * STAGE_BYTES;
          const uint32_t ys = xs + X_BYTES;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            uint64_t adesc, bdesc;
            if (!SWAP) {
              adesc = ptx::make_sdesc_sw128(xs + kk * KMAJ_STEP, 16, 1024);
              bdesc = ptx::make_sdesc_sw128(ys + kk * MNMAJ_STEP, MNMAJ_LBO, 1024);
            } else {
              adesc = ptx::make_sdesc_sw128(xs + kk * MNMAJ_STEP, MNMAJ_LBO, 1024);
              bdesc = ptx::make_sdesc_sw128(ys + kk * KMAJ_STEP, 16, 1024);
            }
            ptx::mma_bf16(d_tmem, adesc, bdesc, IDESC, (kb > c.kb0 || kk > 0) ? 1u : 0u);
          }
          any = true;
          ptx::mma_commit(ptx::smem_u32(&empty[stage]));   // frees the slot when these MMAs finish
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        ptx::mma_commit(ptx::smem_u32(&tfull[acc]));        // accumulator complete
        if (seq == 0) trace_stamp(trace, kTrFirstMmaDone);
        if (++acc == ACC) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (!ok) {
        raise_error(p.err, abort_flag, kErrMmaWait);
        if (any) {
          ptx::mma_commit(ptx::smem_u32(drain));
          ptx::mbar_wait(ptx::smem_u32(drain), 0, nullptr);
        }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue
    const int q = warp & 3;                 // tensor-memory lane quarter of this warp
    const int r = q * 32 + lane;            // accumulator row handled by this thread
    const int et = threadIdx.x - 64;        // 0 .. 127
    int acc = 0;
    uint32_t acc_phase = 0;
    uint32_t red_it = 0;                    // cluster reductions done by this CTA
    uint32_t stg = 0;                       // staging buffers used (TMA-store epilogue)
    const uint32_t staging = tiles_base + STAGES * STAGE_BYTES;
    bool waited = !epi_defer;               // past the wait for the previous grid
    auto wait_prev = [&]() {
      if (waited) return;
      ptx::griddep_wait();
      waited = true;
      if (et == 0) trace_stamp(trace, kTrSetup);
    };
    for (int seq = 0;; ++seq) {
      const int slot = seq % kUnitRing;
      int u = int(blockIdx.x) + seq * int(gridDim.x);     // static round-robin
      if (p.dyn) {
        bool okq = ptx::mbar_wait(ptx::smem_u32(&ufull[slot]), uint32_t(seq / kUnitRing) & 1u, abort_flag, wlim);
        okq = ptx::named_bar_and(1, 128, okq);
        if (!okq) {
          if (et == 0) raise_error(p.err, abort_flag, kErrEpilogueWait);
          break;
        }
        u = uring[slot];
      }
      if (u >= p.total_units) break;
      const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
      // the GEMM's output description, read from the parameter block while
      // the accumulator is still being computed
      const GemmWork w = p.g[c.g];
      const CView cv = c_view<OUT_BF16>(w, c.b);
      bool released = false;                // accumulator already handed back
      bool ok = ptx::mbar_wait(ptx::smem_u32(&tfull[acc]), acc_phase, abort_flag, wlim);
      ok = ptx::named_bar_and(1, 128, ok);
      if (!ok) {
        if (et == 0) raise_error(p.err, abort_flag, kErrEpilogueWait);
        break;
      }
      // every epilogue thread has read the unit's slot (the barrier above)
      if (p.dyn && et == 0) ptx::mbar_arrive(ptx::smem_u32(&uempty[slot]));
      ptx::tc_fence_after();
      const bool first_unit = (seq == 0);
      if (first_unit && et == 0) trace_stamp(trace, kTrFirstAcc);
      const int m0 = c.tm * TILE_M;
      const int n0 = c.tn * TILE_N;
      const uint32_t taddr = tmem_base + (uint32_t(q * 32) << 16) + uint32_t(acc * MMA_N);
      // this CTA's last tile with nothing but tensor stores: the operand
      // ring is idle (every MMA done, no load left) and stages all of it
      // (two-per-SM kinds too, where their ring holds the tile: they keep no
      // staging buffers and store their other tiles directly)
      static_assert(!EPI_TMA || kWideFits, "the ring holds a whole tile");
      const bool wide = kWideFits && w.split == 1 && w.c_tma && p.dyn == nullptr &&
                        u + int(gridDim.x) >= p.total_units;
      // the cluster reductions on chip exchange partials through shared
      // memory only and wait just before their stores
      const bool onchip = kPartFitsRing && p.cluster > 0 && p.total_units == int(gridDim.x);
      if (wide) {
        store_tile_tma<MMA_N, OUT_BF16, true>(&p.tmap_c[c.g], tiles_base, stg, taddr, r, et, m0, n0, c.b);
        wait_prev();
        issue_tile_wide<MMA_N, OUT_BF16>(&p.tmap_c[c.g], tiles_base, et, m0, n0, c.b);
      } else if (!(w.split > 1 && (push_on || onchip))) {
        wait_prev();
      }
      if (wide) {
      } else if (EPI_TMA && w.split == 1 && w.c_tma) {
        store_tile_tma<MMA_N, OUT_BF16>(&p.tmap_c[c.g], staging, stg, taddr, r, et, m0, n0, c.b);
      } else if (w.split == 1) {
#pragma unroll 1
        for (int c0 = 0; c0 < MMA_N; c0 += 32) {
          uint32_t raw[32];
          __syncwarp();
          ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
          ptx::tmem_ld_wait();
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(raw[j]);
          store_chunk<SWAP, OUT_BF16>(cv, m0, n0, r, c0, v);
        }
      } else if (push_on) {
        // ---- cluster split-K, pushed: one unit per CTA.  Row r of the
        // accumulator belongs to the CTA of rank r / (128/S).  The partial
        // goes into the ring (free once the accumulator is complete) as S
        // slices of 128/S rows, 32 columns at a time; as soon as a chunk is
        // staged, one bulk copy per peer sends it that chunk of its slice,
        // counted on the peer's receive barrier, while the next chunk is read
        // out of tensor memory.  Then wait until every peer's copies of this
        // CTA's slice have landed and reduce the S slices from local shared
        // memory.  The cluster barrier at kernel exit keeps every source
        // buffer alive until its copies have landed.
        const int S = w.split;
        const int R = 128 / S;
        const int d = r / R;                   // rank that reduces this row
        const int rr = r - d * R;              // row within that rank's slice
        const uint32_t slot_bytes = uint32_t(R * MMA_N * 4);
        const uint32_t stage_row = tiles_base + uint32_t(d) * slot_bytes;
        const uint32_t recv_slots = tiles_base + uint32_t(STAGES * STAGE_BYTES);
        const uint32_t chunk_bytes = uint32_t(R * 128);
        // the copy this thread issues (threads 0 .. S-1 other than this CTA's rank)
        const bool sender = et < S && et != c.s;
        const uint32_t send_src = tiles_base + uint32_t(et) * slot_bytes;
        const uint32_t send_dst =
            sender ? ptx::map_to_rank(recv_slots + uint32_t(c.s < et ? c.s : c.s - 1) * slot_bytes, uint32_t(et)) : 0u;
        const uint32_t send_bar = sender ? ptx::map_to_rank(ptx::smem_u32(recvbar), uint32_t(et)) : 0u;
#pragma unroll 1
        for (int c0 = 0; c0 < MMA_N; c0 += 32) {
          uint32_t raw[32];
          __syncwarp();
          ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4)
            ptx::st_shared_v4(stage_row + push_offset(rr, c0 / 4 + j4, R), raw[4 * j4], raw[4 * j4 + 1],
                              raw[4 * j4 + 2], raw[4 * j4 + 3]);
          ptx::fence_proxy_async_smem();                 // the chunk visible to the bulk copies
          ptx::named_bar_sync(1, 128);
          if (sender) {
            const uint32_t off = uint32_t(c0 / 32) * chunk_bytes;
            ptx::bulk_copy_to_peer(send_dst + off, send_src + off, chunk_bytes, send_bar);
          }
        }
        ptx::tc_fence_before();
        ptx::mbar_arrive(ptx::smem_u32(&tempty[acc]));   // accumulator no longer needed
        released = true;
        if (first_unit && et == 0) trace_stamp(trace, kTrPartials);
        bool ok2 = ptx::mbar_wait_cluster(ptx::smem_u32(recvbar), 0, abort_flag, wlim);
        ok2 = ptx::named_bar_and(1, 128, ok2);
        if (!ok2) {
          if (et == 0) raise_error(p.err, abort_flag, kErrClusterWait);
          break;
        }
        if (first_unit && et == 0) trace_stamp(trace, kTrArrived);
        wait_prev();
        const uint32_t own_slot = tiles_base + uint32_t(c.s) * slot_bytes;
        switch (S) {
          case 2: reduce_slice_pushed<MMA_N, 2, SWAP, OUT_BF16>(cv, own_slot, recv_slots, c.s, m0, n0, et); break;
          case 4: reduce_slice_pushed<MMA_N, 4, SWAP, OUT_BF16>(cv, own_slot, recv_slots, c.s, m0, n0, et); break;
          case 8: reduce_slice_pushed<MMA_N, 8, SWAP, OUT_BF16>(cv, own_slot, recv_slots, c.s, m0, n0, et); break;
          default: break;
        }
      } else if (onchip) {
        // ---- cluster split-K on chip: one unit per CTA, so the ring's shared
        // memory is free once the accumulator is complete.  Publish the fp32
        // partial there, signal every peer, wait for all S partials, reduce
        // this CTA's rows reading the peers' shared memory.  The cluster
        // barrier at kernel exit keeps every CTA resident until its peers are
        // done reading.
        const uint32_t part_smem = tiles_base;
#pragma unroll 1
        for (int c0 = 0; c0 < MMA_N; c0 += 32) {
          uint32_t raw[32];
          __syncwarp();
          ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4)
            ptx::st_shared_v4(part_smem + part_offset<MMA_N>(r, c0 / 4 + j4), raw[4 * j4], raw[4 * j4 + 1],
                              raw[4 * j4 + 2], raw[4 * j4 + 3]);
        }
        ptx::tc_fence_before();
        ptx::mbar_arrive(ptx::smem_u32(&tempty[acc]));   // accumulator no longer needed
        released = true;
        ptx::fence_acq_rel_cluster();
        ptx::named_bar_sync(1, 128);
        const uint32_t rb = ptx::smem_u32(&redbar[red_it & 1]);
        if (et == 0) {
          if (first_unit) trace_stamp(trace, kTrPartials);
          for (int q2 = 0; q2 < w.split; ++q2) ptx::mbar_arrive_remote_release(ptx::map_to_rank(rb, uint32_t(q2)));
        }
        bool ok2 = ptx::mbar_wait_cluster(rb, (red_it >> 1) & 1, abort_flag, wlim);
        ok2 = ptx::named_bar_and(1, 128, ok2);
        ++red_it;
        if (!ok2) {
          if (et == 0) raise_error(p.err, abort_flag, kErrClusterWait);
          break;
        }
        if (first_unit && et == 0) trace_stamp(trace, kTrArrived);
        wait_prev();
        switch (w.split) {
          case 2: reduce_slice_dsmem<MMA_N, 2, SWAP, OUT_BF16>(cv, part_smem, c.s, m0, n0, et); break;
          case 4: reduce_slice_dsmem<MMA_N, 4, SWAP, OUT_BF16>(cv, part_smem, c.s, m0, n0, et); break;
          case 8: reduce_slice_dsmem<MMA_N, 8, SWAP, OUT_BF16>(cv, part_smem, c.s, m0, n0, et); break;
          default: break;
        }
      } else {
        // partial tile layout: [chunk][float4 index j4][row r] -> coalesced per warp
        constexpr int TILE_F4 = 128 * MMA_N / 4;
        float4* part_base = reinterpret_cast<float4*>(w.ws_part);
        float4* mine = part_base + size_t(c.tile * w.split + c.s) * TILE_F4;
#pragma unroll 1
        for (int c0 = 0; c0 < MMA_N; c0 += 32) {
          uint32_t raw[32];
          __syncwarp();
          ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4)
            mine[((c0 / 4) + j4) * 128 + r] =
                make_float4(__uint_as_float(raw[4 * j4]), __uint_as_float(raw[4 * j4 + 1]),
                            __uint_as_float(raw[4 * j4 + 2]), __uint_as_float(raw[4 * j4 + 3]));
        }
        __threadfence();
        if (p.cluster > 0) {
          // ---- cluster split-K: the S splits of this tile are the S CTAs of
          // this cluster.  Publish the partial, signal every peer, wait for
          // all S partials, then reduce this CTA's 1/S of the tile's rows.
          ptx::tc_fence_before();
          ptx::mbar_arrive(ptx::smem_u32(&tempty[acc]));   // accumulator no longer needed
          released = true;
          ptx::named_bar_sync(1, 128);
          const uint32_t rb = ptx::smem_u32(&redbar[red_it & 1]);
          if (et == 0) {
            if (first_unit) trace_stamp(trace, kTrPartials);
            for (int q2 = 0; q2 < w.split; ++q2) ptx::mbar_arrive_remote_release(ptx::map_to_rank(rb, uint32_t(q2)));
          }
          bool ok2 = ptx::mbar_wait_cluster(rb, (red_it >> 1) & 1, abort_flag, wlim);
          ok2 = ptx::named_bar_and(1, 128, ok2);
          ++red_it;
          if (!ok2) {
            if (et == 0) raise_error(p.err, abort_flag, kErrClusterWait);
            break;
          }
          if (first_unit && et == 0) trace_stamp(trace, kTrArrived);
          const float4* tile_parts = part_base + size_t(c.tile * w.split) * TILE_F4;
          switch (w.split) {
            case 2: reduce_slice<MMA_N, 2, SWAP, OUT_BF16>(cv, tile_parts, c.s, m0, n0, et); break;
            case 4: reduce_slice<MMA_N, 4, SWAP, OUT_BF16>(cv, tile_parts, c.s, m0, n0, et); break;
            case 8: reduce_slice<MMA_N, 8, SWAP, OUT_BF16>(cv, tile_parts, c.s, m0, n0, et); break;
            default: break;
          }
        } else {
        ptx::named_bar_sync(1, 128);
        if (et == 0) {
          if (first_unit) trace_stamp(trace, kTrPartials);
          const uint32_t old = atomicAdd(&w.ws_cnt[c.tile], 1u);
          *last_flag = (old == uint32_t(w.split - 1)) ? 1 : 0;
          if (first_unit) trace_stamp(trace, kTrArrived);
        }
        ptx::named_bar_sync(1, 128);
        if (*last_flag) {
          __threadfence();
#pragma unroll 1
          for (int c0 = 0; c0 < MMA_N; c0 += 32) {
            uint32_t raw[32];
            __syncwarp();
            ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
            ptx::tmem_ld_wait();
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.0f;
            // two splits' partials are loaded before either is added, so their
            // loads are in flight together; the sum runs in split order
            // 0, 1, ..., S-1 (the own split's values come from tensor memory)
#pragma unroll 1
            for (int s2 = 0; s2 < w.split; s2 += 2) {
              const bool has_b = s2 + 1 < w.split;
              float4 ta[8], tb[8];
              const float4* pa = part_base + size_t(c.tile * w.split + s2) * TILE_F4;
              const float4* pb = part_base + size_t(c.tile * w.split + s2 + 1) * TILE_F4;
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                const float4 own = make_float4(__uint_as_float(raw[4 * j4]), __uint_as_float(raw[4 * j4 + 1]),
                                               __uint_as_float(raw[4 * j4 + 2]), __uint_as_float(raw[4 * j4 + 3]));
                ta[j4] = (s2 == c.s) ? own : __ldcg(&pa[((c0 / 4) + j4) * 128 + r]);
                tb[j4] = (!has_b || s2 + 1 == c.s) ? own : __ldcg(&pb[((c0 / 4) + j4) * 128 + r]);
              }
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                v[4 * j4] += ta[j4].x;
                v[4 * j4 + 1] += ta[j4].y;
                v[4 * j4 + 2] += ta[j4].z;
                v[4 * j4 + 3] += ta[j4].w;
              }
              if (has_b) {
#pragma unroll
                for (int j4 = 0; j4 < 8; ++j4) {
                  v[4 * j4] += tb[j4].x;
                  v[4 * j4 + 1] += tb[j4].y;
                  v[4 * j4 + 2] += tb[j4].z;
                  v[4 * j4 + 3] += tb[j4].w;
                }
              }
            }
            store_chunk<SWAP, OUT_BF16>(cv, m0, n0, r, c0, v);
          }
          if (et == 0) w.ws_cnt[c.tile] = 0u;     // leave the counter zeroed for the next run
        }
        }
      }
      if (first_unit && et == 0) trace_stamp(trace, kTrFirstStore);
      if (!released) {
        ptx::tc_fence_before();
        ptx::mbar_arrive(ptx::smem_u32(&tempty[acc]));
      }
      if (++acc == ACC) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    // tensor stores must have read the staging buffers before the CTA leaves
    // (their writes to C complete with the grid)
    if ((EPI_TMA || kWideFits) && et == 0) ptx::bulk_wait_group_read<0>();
  }

  __syncthreads();
  if (threadIdx.x == 0) {
    trace_stamp(trace, kTrEnd);
    if (trace) trace[blockIdx.x * kTracePerCta + kTrUnits] = *units_taken;
    if (p.dyn) {
      // every CTA has stopped taking units once all have counted themselves
      // out: the last one zeroes the counters for the next launch
      __threadfence();
      if (atomicAdd(p.dyn + 1, 1u) == gridDim.x - 1) {
        p.dyn[0] = 0u;
        p.dyn[1] = 0u;
        __threadfence();
      }
    }
  }
  // no CTA of a cluster leaves while a peer may still signal its barriers
  // (every role's waits are bounded, so every CTA gets here)
  if (p.cluster > 0) ptx::cluster_sync_all();
  if (warp == 1) {
    __syncwarp();
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

}  // namespace goldy

// GO-Kernel over CTA pairs: 256 x 256 output tiles with tcgen05.mma.cta_group::2.
//
// Same GEMM as go_gemm_kernel (Sec. 2.1.2, C = A * B, fp32 accumulation), for
// compute-bound shapes.  A cluster of two CTAs on neighbouring SMs works on one
// 256 x 256 tile at a time: CTA r (r = 0, 1) loads rows 128r .. 128r+127 of the
// tile's A panel and columns 128r .. 128r+127 of its B panel into its own
// shared memory, the even CTA issues one 256 x 256 x 16 MMA per K step that
// reads both CTAs' operands, and each CTA's tensor memory receives its 128
// rows of the accumulator.  Per K block each SM therefore takes in 32 KB of
// operands for 128 x 256 x 64 multiply-adds — two thirds of what the
// single-CTA 128 x 256 tile needs — which keeps the tensor cores fed from L2.
//
// Roles per CTA (192 threads): warp 0 lane 0 loads (both CTAs; the odd CTA's
// loads complete on the even CTA's barrier), warp 1 allocates tensor memory
// jointly with the peer and, in the even CTA, issues the MMAs and commits
// (multicast to both CTAs' barriers), warps 2-5 drain the CTA's own half of
// the accumulator.  Units (256 x 256 tiles, or with a K split S, S K-ranges
// of a tile) go to pairs round-robin; both CTAs of a pair walk the same
// sequence.  With S > 1 each CTA publishes its 128 x 256 fp32 partial to the
// workspace and the last split to arrive for a tile half sums the S partials
// in split order and stores C.  Every wait is bounded; before leaving,
// each CTA waits (bounded) until every arrival the peer owes its barriers has
// landed, then the pair meets at a cluster barrier.
#pragma once

#include "go_kernel.cuh"

namespace goldy {

template <bool OUT_BF16, int MAXG>
__global__ void __launch_bounds__(192, 1) go_gemm_pair_kernel(const __grid_constant__ LaunchParams<MAXG> p) {
  constexpr int STAGES = 6;
  constexpr int ACC = 2;
  constexpr int HALF_N = 128;                        // B columns held per CTA
  constexpr int A_BYTES = 128 * 64 * 2;              // 128 rows of A x 64 K
  constexpr int B_BYTES = HALF_N * 64 * 2;           // 128 columns of B x 64 K
  constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  constexpr uint32_t TMEM_COLS = 512;                // 2 accumulators x 256 fp32 columns
  constexpr uint32_t IDESC = ptx::make_idesc_bf16(256, 256, 0, 1);
  constexpr uint32_t KMAJ_STEP = 32;
  constexpr uint32_t MNMAJ_STEP = 2048;
  constexpr uint32_t MNMAJ_LBO = 64 * 128;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int STAGING_BYTES = 2 * 16384;            // TMA-store epilogue buffers
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES + STAGING_BYTES);
  uint64_t* full = bars;                    // used in the even CTA: both CTAs' loads complete here
  uint64_t* empty = bars + STAGES;          // each CTA: its slot was consumed by the pair MMA
  uint64_t* tfull = bars + 2 * STAGES;      // each CTA: its half of the accumulator is ready
  uint64_t* tempty = bars + 2 * STAGES + ACC;  // even CTA: both halves were drained (2 arrivals)
  uint64_t* drain = bars + 2 * STAGES + 2 * ACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);   // split-K: last arriver
  UnitTable* utab = reinterpret_cast<UnitTable*>(tmem_slot + 4);   // see go_gemm_kernel
  static_assert((2 * STAGES + 2 * ACC + 1) * 8 + 16 + MAXG * int(sizeof(UnitTable)) <= 1024, "barrier area");
  const int n_gemms = p.n_gemms;

  const uint32_t tiles_base = ptx::smem_u32(smem);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank() & 1u;
  const bool lead = rank == 0;
  const int pair = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;
  unsigned long long* const trace = p.trace;
  ptx::griddep_launch_dependents();   // see go_gemm_kernel

  if (threadIdx.x == 0) {
    trace_stamp(trace, kTrStart);
    if (trace) {
      uint32_t sm;
      asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
      trace[blockIdx.x * kTracePerCta + kTrSm] = sm;
      trace[blockIdx.x * kTracePerCta + kTrGrid] = gridDim.x;
      trace[blockIdx.x * kTracePerCta + kTrCta] = blockIdx.x;
    }
    for (int g = 0; g < p.n_gemms; ++g) {
      ptx::prefetch_tensormap(&p.tmap_a[g]);
      ptx::prefetch_tensormap(&p.tmap_b[g]);
      if (p.g[g].c_tma) ptx::prefetch_tensormap(&p.tmap_c[g]);
    }
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(ptx::smem_u32(&full[s]), 1);
      ptx::mbar_init(ptx::smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < ACC; ++a) {
      ptx::mbar_init(ptx::smem_u32(&tfull[a]), 1);
      ptx::mbar_init(ptx::smem_u32(&tempty[a]), 2);
    }
    ptx::mbar_init(ptx::smem_u32(drain), 1);
    *abort_flag = 0;
    *last_flag = 0;
    ptx::fence_barrier_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc_pair(ptx::smem_u32(tmem_slot), TMEM_COLS);
    ptx::tmem_relinquish_pair();
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
  ptx::cluster_sync_all();                  // the peer's barriers and tensor memory are ready
  ptx::tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint64_t wlim = p.wait_ns ? p.wait_ns : ptx::kWaitLimitNs;
  // global memory only after the previous grid is done; in early mode the
  // load and MMA roles go ahead (see go_gemm_kernel) and the epilogue waits
  const bool early = p.early_loads != 0 && warp < 2;
  // in early mode the epilogue waits where it first writes global memory
  // (below); a CTA's last tile is staged in the idle ring before that wait
  const bool epi_defer = p.early_loads != 0 && warp >= 2;
  if (!early && !epi_defer) ptx::griddep_wait();
  if (threadIdx.x == 64 && !epi_defer) trace_stamp(trace, kTrSetup);   // the first epilogue thread waits

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ producer
      int stage = 0;
      uint32_t phase = 0, issued = 0, last_phase = 0;
      bool ok = true;
      for (int u = pair; ok && u < p.total_units; u += n_pairs) {
        const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
        const void* ta = &p.tmap_a[c.g];
        const void* tb = &p.tmap_b[c.g];
        const int m0 = c.tm * 256 + int(rank) * 128;
        const int n0 = c.tn * 256 + int(rank) * HALF_N;
        for (int kb = c.kb0; kb < c.kb1; ++kb) {
          // only a slot filled before is waited for (see go_gemm_kernel)
          if ((issued >> stage & 1) && !ptx::mbar_wait(ptx::smem_u32(&empty[stage]), phase ^ 1, abort_flag, wlim)) {
            ok = false;
            break;
          }
          const uint32_t fb_local = ptx::smem_u32(&full[stage]);
          const uint32_t fb = ptx::map_to_rank(fb_local, 0);      // the even CTA's barrier
          if (lead) ptx::mbar_arrive_expect_tx(fb_local, 2 * STAGE_BYTES);
          const uint32_t xs = tiles_base + stage * STAGE_BYTES;
          const uint32_t ys = xs + A_BYTES;
          const int k0 = kb * 64;
          ptx::tma_load_3d_pair(xs, ta, fb, k0, m0, c.b);
          ptx::tma_load_3d_pair(ys, tb, fb, n0, k0, c.b);
          ptx::tma_load_3d_pair(ys + 8192, tb, fb, n0 + 64, k0, c.b);
          if (issued == 0) trace_stamp(trace, kTrFirstLoad);
          issued |= 1u << stage;
          last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) raise_error(p.err, abort_flag, kErrProducerWait);
      // every slot this CTA filled must have been released by the pair MMA
      // (so the even CTA's commits to this CTA's barriers have landed, and
      // the peer's loads into the even CTA's slots are done) before leaving
      const uint64_t t0 = ptx::global_timer();
      for (int s = 0; s < STAGES; ++s) {
        if (!(issued >> s & 1)) continue;
        const uint32_t bar = ptx::smem_u32(&empty[s]);
        const uint32_t par = (last_phase >> s) & 1;
        while (!ptx::mbar_try_wait(bar, par)) {
          if (ptx::global_timer() - t0 > wlim) {
            raise_error(p.err, abort_flag, kErrProducerWait);
            break;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && lead) {
      // ------------------------------------------------- MMA issuer (even CTA)
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0, acc_used = 0;
      bool ok = true, any = false;
      for (int u = pair; ok && u < p.total_units; u += n_pairs) {
        const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
        // both CTAs drained this accumulator (the odd CTA signals with a
        // cluster-scope release, so wait with a cluster-scope acquire); the
        // first use of an accumulator needs no wait
        if ((acc_used >> acc & 1) &&
            !ptx::mbar_wait_cluster(ptx::smem_u32(&tempty[acc]), acc_phase ^ 1, abort_flag, wlim)) {
          ok = false;
          break;
        }
        acc_used |= 1u << acc;
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + uint32_t(acc * 256);
        for (int kb = c.kb0; kb < c.kb1; ++kb) {
          if (!ptx::mbar_wait(ptx::smem_u32(&full[stage]), phase, abort_flag, wlim)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          if (!any) trace_stamp(trace, kTrFirstFull);
          const uint32_t xs = tiles_base + stage * STAGE_BYTES;
          const uint32_t ys = xs + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t adesc = ptx::make_sdesc_sw128(xs + kk * KMAJ_STEP, 16, 1024);
            const uint64_t bdesc = ptx::make_sdesc_sw128(ys + kk * MNMAJ_STEP, MNMAJ_LBO, 1024);
            ptx::mma_bf16_pair(d_tmem, adesc, bdesc, IDESC, (kb > c.kb0 || kk > 0) ? 1u : 0u);
          }
          any = true;
          ptx::mma_commit_pair_multicast(ptx::smem_u32(&empty[stage]), 0x3);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        ptx::mma_commit_pair_multicast(ptx::smem_u32(&tfull[acc]), 0x3);
        if (u == pair) trace_stamp(trace, kTrFirstMmaDone);
        if (++acc == ACC) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (!ok) {
        raise_error(p.err, abort_flag, kErrMmaWait);
        if (any) {
          ptx::mma_commit_pair_multicast(ptx::smem_u32(drain), 0x1);
          ptx::mbar_wait(ptx::smem_u32(drain), 0, nullptr);
        }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int et = threadIdx.x - 64;
    int acc = 0;
    uint32_t acc_phase = 0;
    uint32_t stg = 0;
    const uint32_t staging = tiles_base + STAGES * STAGE_BYTES;
    bool waited = !epi_defer;               // past the wait for the previous grid
    auto wait_prev = [&]() {
      if (waited) return;
      ptx::griddep_wait();
      waited = true;
      if (et == 0) trace_stamp(trace, kTrSetup);
    };
    for (int u = pair; u < p.total_units; u += n_pairs) {
      const UnitCoord c = decode_unit_tab(utab, n_gemms, u);
      const GemmWork w = p.g[c.g];                 // read while the accumulator is computed
      const CView cv = c_view<OUT_BF16>(w, c.b);
      bool ok = ptx::mbar_wait(ptx::smem_u32(&tfull[acc]), acc_phase, abort_flag, wlim);
      ok = ptx::named_bar_and(1, 128, ok);
      if (!ok) {
        if (et == 0) raise_error(p.err, abort_flag, kErrEpilogueWait);
        break;
      }
      ptx::tc_fence_after();
      const bool first_unit = (u == pair);
      if (first_unit && et == 0) trace_stamp(trace, kTrFirstAcc);
      const int m0 = c.tm * 256 + int(rank) * 128;
      const int n0 = c.tn * 256;
      const uint32_t taddr = tmem_base + (uint32_t(q * 32) << 16) + uint32_t(acc * 256);
      // this CTA's last tile: every MMA has completed (the accumulator is
      // ready) and no load is left, so the operand ring is idle and stages
      // the whole tile (128 KB fp32 / 64 KB bf16 of its 192 KB) before the
      // wait; only the stores follow it
      const bool wide = w.split == 1 && w.c_tma && u + n_pairs >= p.total_units;
      static_assert(STAGES * STAGE_BYTES >= 256 * 512, "the ring holds a whole tile half");
      if (wide) {
        store_tile_tma<256, OUT_BF16, true>(&p.tmap_c[c.g], tiles_base, stg, taddr, r, et, m0, n0, c.b);
        wait_prev();
        issue_tile_wide<256, OUT_BF16>(&p.tmap_c[c.g], tiles_base, et, m0, n0, c.b);
      } else {
        wait_prev();
      }
      if (wide) {
      } else if (w.split > 1) {
        // ---- split-K: this CTA publishes its fp32 partial (its 128 rows of
        // the 256 x 256 tile, layout [chunk][float4][row]) to the workspace
        // and counts itself in; the last of the S splits to arrive for this
        // tile half sums the S partials in split order 0, 1, ..., S-1 (its
        // own from tensor memory) and stores C, then zeroes the counter.  No
        // CTA waits for another.
        constexpr int TILE_F4 = 128 * 256 / 4;
        float4* part_base = reinterpret_cast<float4*>(w.ws_part);
        const size_t half = size_t(c.tile) * 2 + rank;
        float4* mine = part_base + (half * size_t(w.split) + size_t(c.s)) * TILE_F4;
#pragma unroll 1
        for (int c0 = 0; c0 < 256; c0 += 32) {
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
        ptx::named_bar_sync(1, 128);
        if (et == 0) {
          const uint32_t old = atomicAdd(&w.ws_cnt[half], 1u);
          *last_flag = (old == uint32_t(w.split - 1)) ? 1 : 0;
        }
        ptx::named_bar_sync(1, 128);
        if (*last_flag) {
          __threadfence();
          const float4* parts = part_base + half * size_t(w.split) * TILE_F4;
#pragma unroll 1
          for (int c0 = 0; c0 < 256; c0 += 32) {
            uint32_t raw[32];
            __syncwarp();
            ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
            ptx::tmem_ld_wait();
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.0f;
#pragma unroll 1
            for (int s2 = 0; s2 < w.split; ++s2) {
              float4 t[8];
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4)
                t[j4] = (s2 == c.s) ? make_float4(__uint_as_float(raw[4 * j4]), __uint_as_float(raw[4 * j4 + 1]),
                                                   __uint_as_float(raw[4 * j4 + 2]), __uint_as_float(raw[4 * j4 + 3]))
                                    : __ldcg(&parts[size_t(s2) * TILE_F4 + ((c0 / 4) + j4) * 128 + r]);
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                v[4 * j4] += t[j4].x;
                v[4 * j4 + 1] += t[j4].y;
                v[4 * j4 + 2] += t[j4].z;
                v[4 * j4 + 3] += t[j4].w;
              }
            }
            store_chunk<false, OUT_BF16>(cv, m0, n0, r, c0, v);
          }
          if (et == 0) w.ws_cnt[half] = 0u;     // leave the counter zeroed for the next run
        }
      } else if (w.c_tma) {
        store_tile_tma<256, OUT_BF16>(&p.tmap_c[c.g], staging, stg, taddr, r, et, m0, n0, c.b);
      } else {
#pragma unroll 1
        for (int c0 = 0; c0 < 256; c0 += 32) {
          uint32_t raw[32];
          __syncwarp();
          ptx::tmem_ld_32x32b_x32(taddr + c0, raw);
          ptx::tmem_ld_wait();
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(raw[j]);
          store_chunk<false, OUT_BF16>(cv, m0, n0, r, c0, v);
        }
      }
      if (first_unit && et == 0) trace_stamp(trace, kTrFirstStore);
      ptx::tc_fence_before();
      ptx::named_bar_sync(1, 128);
      if (et == 0) {
        // this CTA's half of accumulator `acc` is drained: tell the MMA issuer
        ptx::mbar_arrive_remote_release(ptx::map_to_rank(ptx::smem_u32(&tempty[acc]), 0));
      }
      if (++acc == ACC) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    // the tensor stores must have read their shared-memory sources before
    // the CTA leaves; their writes to C complete with the grid, which is
    // what a dependent launch's griddepcontrol.wait waits for
    if (et == 0) ptx::bulk_wait_group_read<0>();
  }

  __syncthreads();
  if (threadIdx.x == 0) {
    trace_stamp(trace, kTrEnd);
    if (trace) {
      int n = 0;
      for (int u = pair; u < p.total_units; u += n_pairs) ++n;
      trace[blockIdx.x * kTracePerCta + kTrUnits] = n;
    }
  }
  ptx::cluster_sync_all();                  // no CTA of the pair leaves while the other may still signal it
  if (warp == 1) {
    __syncwarp();
    ptx::tc_fence_after();
    ptx::tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

}  // namespace goldy

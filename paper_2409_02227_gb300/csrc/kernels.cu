// Instantiates the GO-Kernel template for one kind (compile with
// -DGOLDY_KIND=k, k in 0 .. kNumKinds-1), both output dtypes, and both launch
// forms (one GEMM per launch, or up to kMaxFused GEMMs).  One object per kind
// keeps the build parallel.
#include "go_kernel.cuh"
#include "go_kernel_pair.cuh"
#include "goldy_internal.h"

#ifndef GOLDY_KIND
#error "compile kernels.cu with -DGOLDY_KIND=<kind index>"
#endif

#define GOLDY_CAT2(a, b) a##b
#define GOLDY_CAT(a, b) GOLDY_CAT2(a, b)

namespace goldy {

// Inside a template, `if constexpr` discards the other family entirely.
template <int KIND>
const void* select_kernel(int out_bf16, int fused) {
  constexpr KindInfo k = kKinds[KIND];
  constexpr bool swap = k.swap_ab != 0;
  static_assert(k.pair != 0 || PushRecv<k.mma_n, k.ctas_per_sm>::bytes == push_recv_bytes(k),
                "host and kernel agree on the pushed reduction's receive slots");
  static_assert(smem_bytes(k) <= 232448, "shared memory per CTA");
  if constexpr (k.pair != 0) {
    if (fused)
      return out_bf16 ? reinterpret_cast<const void*>(&go_gemm_pair_kernel<true, kMaxFused>)
                      : reinterpret_cast<const void*>(&go_gemm_pair_kernel<false, kMaxFused>);
    return out_bf16 ? reinterpret_cast<const void*>(&go_gemm_pair_kernel<true, 1>)
                    : reinterpret_cast<const void*>(&go_gemm_pair_kernel<false, 1>);
  } else {
    if (fused) {
      if (out_bf16)
        return reinterpret_cast<const void*>(
            &go_gemm_kernel<k.mma_n, swap, k.stages, k.acc_stages, true, kMaxFused, k.ctas_per_sm, epi_tma(k)>);
      return reinterpret_cast<const void*>(
          &go_gemm_kernel<k.mma_n, swap, k.stages, k.acc_stages, false, kMaxFused, k.ctas_per_sm, epi_tma(k)>);
    }
    if (out_bf16)
      return reinterpret_cast<const void*>(
          &go_gemm_kernel<k.mma_n, swap, k.stages, k.acc_stages, true, 1, k.ctas_per_sm, epi_tma(k)>);
    return reinterpret_cast<const void*>(
        &go_gemm_kernel<k.mma_n, swap, k.stages, k.acc_stages, false, 1, k.ctas_per_sm, epi_tma(k)>);
  }
}

const void* GOLDY_CAT(kernel_fn_k, GOLDY_KIND)(int out_bf16, int fused) {
  return select_kernel<GOLDY_KIND>(out_bf16, fused);
}

}  // namespace goldy

// Instantiates the GO-Kernel template for one kind (compile with
// -DGOLDY_KIND=k, k in 0 .. kNumKinds-1), both output dtypes, and both launch
// forms (one GEMM per launch, or up to kMaxFused GEMMs).  One object per kind
// keeps the build parallel.
#include "go_kernel.cuh"
#include "goldy_internal.h"

#ifndef GOLDY_KIND
#error "compile kernels.cu with -DGOLDY_KIND=<kind index>"
#endif

#define GOLDY_CAT2(a, b) a##b
#define GOLDY_CAT(a, b) GOLDY_CAT2(a, b)

namespace goldy {

namespace {
constexpr KindInfo kK = kKinds[GOLDY_KIND];
constexpr bool kSwap = kK.swap_ab != 0;
}  // namespace

const void* GOLDY_CAT(kernel_fn_k, GOLDY_KIND)(int out_bf16, int fused) {
  if (fused) {
    if (out_bf16)
      return reinterpret_cast<const void*>(
          &go_gemm_kernel<kK.mma_n, kSwap, kK.stages, kK.acc_stages, true, kMaxFused, kK.ctas_per_sm>);
    return reinterpret_cast<const void*>(
        &go_gemm_kernel<kK.mma_n, kSwap, kK.stages, kK.acc_stages, false, kMaxFused, kK.ctas_per_sm>);
  }
  if (out_bf16)
    return reinterpret_cast<const void*>(&go_gemm_kernel<kK.mma_n, kSwap, kK.stages, kK.acc_stages, true, 1, kK.ctas_per_sm>);
  return reinterpret_cast<const void*>(&go_gemm_kernel<kK.mma_n, kSwap, kK.stages, kK.acc_stages, false, 1, kK.ctas_per_sm>);
}

}  // namespace goldy

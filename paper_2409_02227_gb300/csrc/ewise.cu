// Element-wise add Z = X + Y: the non-GEMM kernel the paper co-schedules
// with a GEMM (Sec. 7.1: element-wise adds over the GEMM's output size).
//
// HBM-bound: every element is read twice and written once.  Persistent
// grid-stride loop over 16-byte vectors (8 bf16 or 4 fp32 per vector), four
// vectors in flight per thread; kEwiseThreads threads per CTA, at most
// kEwiseCtasPerSm CTAs per SM divided by the grid-cap divisor (the same
// GPU, GPU/2, GPU/4 resource constraint as the GO-Kernels, Sec. 4.2.1).
// Arithmetic: IEEE fp32 addition with round-to-nearest-even; bf16 inputs are
// widened exactly and the fp32 sum is rounded to bf16 (RNE).  Pointers that
// are not 16-byte aligned take the scalar path for the whole array.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "goldy_internal.h"

namespace goldy {
namespace {

constexpr int kUnroll = 4;

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(uint32_t(h) << 16); }

__device__ __forceinline__ uint16_t f32_to_bf16_rne(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

__device__ __forceinline__ uint4 add_vec_bf16(uint4 a, uint4 b) {
  uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w}, out[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = __fadd_rn(bf16_to_f32(uint16_t(av[i] & 0xFFFF)), bf16_to_f32(uint16_t(bv[i] & 0xFFFF)));
    const float hi = __fadd_rn(bf16_to_f32(uint16_t(av[i] >> 16)), bf16_to_f32(uint16_t(bv[i] >> 16)));
    out[i] = uint32_t(f32_to_bf16_rne(lo)) | (uint32_t(f32_to_bf16_rne(hi)) << 16);
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

__device__ __forceinline__ uint4 add_vec_f32(uint4 a, uint4 b) {
  return make_uint4(__float_as_uint(__fadd_rn(__uint_as_float(a.x), __uint_as_float(b.x))),
                    __float_as_uint(__fadd_rn(__uint_as_float(a.y), __uint_as_float(b.y))),
                    __float_as_uint(__fadd_rn(__uint_as_float(a.z), __uint_as_float(b.z))),
                    __float_as_uint(__fadd_rn(__uint_as_float(a.w), __uint_as_float(b.w))));
}

template <bool BF16>
__global__ void __launch_bounds__(kEwiseThreads) ewise_add_kernel(const EwiseParams p) {
  const void* __restrict__ x = p.x;
  const void* __restrict__ y = p.y;
  void* __restrict__ z = p.z;
  const int64_t n = p.n;
  const int vec_ok = p.vec_ok;
  constexpr int kPerVec = BF16 ? 8 : 4;
  const int64_t stride = int64_t(gridDim.x) * kEwiseThreads;
  const int64_t tid = int64_t(blockIdx.x) * kEwiseThreads + threadIdx.x;
  int64_t done = 0;
  if (vec_ok) {
    const uint4* xv = static_cast<const uint4*>(x);
    const uint4* yv = static_cast<const uint4*>(y);
    uint4* zv = static_cast<uint4*>(z);
    const int64_t nv = n / kPerVec;
    int64_t v = tid;
    // four vectors in flight per thread
    for (; v + (kUnroll - 1) * stride < nv; v += kUnroll * stride) {
      uint4 a[kUnroll], b[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        a[u] = __ldcs(xv + v + u * stride);
        b[u] = __ldcs(yv + v + u * stride);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        __stcs(zv + v + u * stride, BF16 ? add_vec_bf16(a[u], b[u]) : add_vec_f32(a[u], b[u]));
    }
    for (; v < nv; v += stride) {
      const uint4 a = __ldcs(xv + v), b = __ldcs(yv + v);
      __stcs(zv + v, BF16 ? add_vec_bf16(a, b) : add_vec_f32(a, b));
    }
    done = nv * kPerVec;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    if (BF16) {
      const uint16_t a = static_cast<const uint16_t*>(x)[i], b = static_cast<const uint16_t*>(y)[i];
      static_cast<uint16_t*>(z)[i] = f32_to_bf16_rne(__fadd_rn(bf16_to_f32(a), bf16_to_f32(b)));
    } else {
      static_cast<float*>(z)[i] = __fadd_rn(static_cast<const float*>(x)[i], static_cast<const float*>(y)[i]);
    }
  }
}

}  // namespace

const void* ewise_kernel_fn(int bf16) {
  return bf16 ? reinterpret_cast<const void*>(&ewise_add_kernel<true>)
              : reinterpret_cast<const void*>(&ewise_add_kernel<false>);
}

}  // namespace goldy

/*
 * Plain fp64 reference GEMM — TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
 * arm may load this library.  The product path (paper_2409_02227_gb300) never
 * links, imports or calls it, and this file shares no code with it.
 *
 * What it computes (Sec. 2.1.2, "GEMM Operation"): a GEMM multiplies A of
 * size M x K with B to give C of size M x N, 2*M*N*K multiplies and adds.
 * The concurrent-GEMM workloads store B as K x N row-major (N contiguous) and
 * A as M x K row-major (K contiguous), both in bfloat16, so
 *
 *     ref[i][j] = sum_{k = 0}^{K-1} A[i][k] * B[k][j]
 *
 * evaluated in double precision, accumulating in increasing k.  Every bf16
 * value is exactly representable in double, every bf16*bf16 product is exact
 * in double (8+8 significant bits), so the only rounding is the fp64
 * accumulation itself.  Build with -ffp-contract=off so that no fused
 * multiply-add changes the summation on any host.
 *
 * Parallelism: OpenMP over output rows only; each output element is still one
 * sequential k-loop, so the result does not depend on the thread count.
 */
#include <stdint.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* bfloat16 is the upper half of an IEEE-754 binary32: decode by shifting the
 * 16 stored bits into the high half of a 32-bit word. */
static double bf16_bits_to_double(uint16_t h) {
  uint32_t u = ((uint32_t)h) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* out[i] = value of the bf16 bit pattern in[i]. */
void oracle_bf16_decode(const uint16_t* in, double* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = bf16_bits_to_double(in[i]);
}

/* Full GEMM: C[i*ldc + j] = sum_k A[i*lda + k] * B[k*ldb + j] for
 * 0 <= i < M, 0 <= j < N.  K == 0 gives zeros. */
void oracle_gemm_bf16(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                      double* C, int64_t ldc, int64_t M, int64_t N, int64_t K) {
  int64_t i;
#pragma omp parallel for schedule(static)
  for (i = 0; i < M; ++i) {
    double* c = C + i * ldc;
    for (int64_t j = 0; j < N; ++j) c[j] = 0.0;
    for (int64_t k = 0; k < K; ++k) {
      const double a = bf16_bits_to_double(A[i * lda + k]);
      const uint16_t* b = B + k * ldb;
      for (int64_t j = 0; j < N; ++j) c[j] += a * bf16_bits_to_double(b[j]);
    }
  }
}

/* Selected rows only: out[r*N + j] = row rows[r] of the product, same
 * arithmetic as oracle_gemm_bf16.  Used when a GEMM is too large to check in
 * full; the sampled entries are still exact reference values. */
void oracle_gemm_bf16_rows(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                           const int64_t* rows, int64_t n_rows, double* out,
                           int64_t N, int64_t K) {
  int64_t r;
#pragma omp parallel for schedule(static)
  for (r = 0; r < n_rows; ++r) {
    const int64_t i = rows[r];
    double* c = out + r * N;
    for (int64_t j = 0; j < N; ++j) c[j] = 0.0;
    for (int64_t k = 0; k < K; ++k) {
      const double a = bf16_bits_to_double(A[i * lda + k]);
      const uint16_t* b = B + k * ldb;
      for (int64_t j = 0; j < N; ++j) c[j] += a * bf16_bits_to_double(b[j]);
    }
  }
}

/* Single entries: out[t] = sum_k A[ii[t]][k] * B[k][jj[t]]. */
void oracle_gemm_bf16_entries(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                              const int64_t* ii, const int64_t* jj, int64_t n, double* out,
                              int64_t K) {
  int64_t t;
#pragma omp parallel for schedule(static)
  for (t = 0; t < n; ++t) {
    double s = 0.0;
    for (int64_t k = 0; k < K; ++k)
      s += bf16_bits_to_double(A[ii[t] * lda + k]) * bf16_bits_to_double(B[k * ldb + jj[t]]);
    out[t] = s;
  }
}

// SIMT GEMM (fp32 FMA) with a separate epilogue pass.  This is the path of the fp32
// models and the cross-check of the tensor-core GEMM; its epilogue semantics are the
// reference for the fused tcgen05 epilogue.
#define ADEPT_TU_ID 2
#include "common.cuh"
#include "kernels.h"
#include "epilogue.cuh"

namespace adept {

// C[r, n] = sum_k A[begin + r, k] * B[n, k] for the rows of the problem's range.
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, int lda, const T* __restrict__ B,
                                                        int ldb, DevRange rows, int N, int K, float* C, int ldc) {
  PDL_ENTRY();
  __shared__ float As[16][64 + 1];
  __shared__ float Bs[16][64 + 1];
  const int rb = rows.b(), M = rows.e() - rb;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  if (m0 >= M) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int i = threadIdx.x; i < 1024; i += 256) {
      const int r = i >> 4, kk = i & 15, gk = k0 + kk;
      As[kk][r] = (m0 + r < M && gk < K) ? to_f(A[(size_t)(rb + m0 + r) * lda + gk]) : 0.f;
      Bs[kk][r] = (n0 + r < N && gk < K) ? to_f(B[(size_t)(n0 + r) * ldb + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Bs[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = m0 + ty * 4 + i;
    if (r >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n < N) C[(size_t)r * ldc + n] = acc[i][j];
    }
  }
}

// Epilogue of one output row (see EpiKind), one thread per 32-column chunk.
template <typename T>
__global__ void epilogue_kernel(Epi e, const float* __restrict__ C, int ldc, DevRange rows, int N) {
  PDL_ENTRY();
  const int rb = rows.b(), M = rows.e() - rb;
  const int r = blockIdx.x;
  if (r >= M) return;
  const int ra = rb + r;
  const float* c = C + (size_t)r * ldc;
  const EpiRow rr = epi_row(e, ra);
  for (int ch = threadIdx.x; ch * 32 < N; ch += blockDim.x) {
    const int c0 = ch * 32;
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = (c0 + j < N) ? c[c0 + j] : 0.f;
    epi_chunk32<T>(e, ra, c0, N, v, rr);
  }
}

void launch_gemm_simt(cudaStream_t st, int dt, const GemmProblem& p, int max_rows, float* scratch) {
  if (max_rows <= 0) return;
  dim3 grid(cdiv(p.N, 64), cdiv(max_rows, 64));
  if (dt == 1) {
    launch_k(gemm_simt_kernel<bf16>, grid, 256, 0, st, (const bf16*)p.A, p.lda, (const bf16*)p.B, p.ldb, p.rows, p.N, p.K,
                                                 scratch, p.N);
    launch_k(epilogue_kernel<bf16>, max_rows, 64, 0, st, p.epi, scratch, p.N, p.rows, p.N);
  } else {
    launch_k(gemm_simt_kernel<float>, grid, 256, 0, st, (const float*)p.A, p.lda, (const float*)p.B, p.ldb, p.rows, p.N,
                                                  p.K, scratch, p.N);
    launch_k(epilogue_kernel<float>, max_rows, 64, 0, st, p.epi, scratch, p.N, p.rows, p.N);
  }
}

ADEPT_KTRACE_ATTACH(simt)

}  // namespace adept

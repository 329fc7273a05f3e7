// SIMT GEMM (fp32 FMA) with a separate epilogue pass.  This is the path of the fp32
// models and the cross-check of the tensor-core GEMM; its epilogue semantics are the
// reference for the fused tcgen05 epilogue.
#include "common.cuh"
#include "kernels.h"

namespace adept {

// C[r, n] = sum_k A[begin + r, k] * B[n, k] for the rows of the problem's range.
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, int lda, const T* __restrict__ B,
                                                        int ldb, DevRange rows, int N, int K, float* C, int ldc) {
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

// Epilogue of one output row (see EpiKind): reads the fp32 accumulators of the row.
template <typename T>
__global__ void epilogue_kernel(Epi e, const float* __restrict__ C, int ldc, DevRange rows, int N) {
  const int rb = rows.b(), M = rows.e() - rb;
  const int r = blockIdx.x;
  if (r >= M) return;
  const int ra = rb + r;
  const float* c = C + (size_t)r * ldc;
  const float* bias = e.bias;
  switch (e.kind) {
    case EPI_F32:
      for (int n = threadIdx.x; n < N; n += blockDim.x) e.out_f32[(size_t)ra * e.ld_f32 + n] = c[n] + (bias ? bias[n] : 0.f);
      return;
    case EPI_ACT:
      for (int n = threadIdx.x; n < N; n += blockDim.x) {
        const float v = apply_act(e.act, c[n] + (bias ? bias[n] : 0.f));
        ((T*)e.out_t)[(size_t)ra * e.ld_t + n] = from_f<T>(v);
        if (e.out_f32) e.out_f32[(size_t)ra * e.ld_f32 + n] = v;
      }
      return;
    case EPI_RESID:
      for (int n = threadIdx.x; n < N; n += blockDim.x)
        e.out_f32[(size_t)ra * e.ld_f32 + n] = e.resid[(size_t)ra * e.ld_resid + n] + c[n] + (bias ? bias[n] : 0.f);
      return;
    case EPI_SWIGLU:
      for (int f = threadIdx.x; f < N / 2; f += blockDim.x) {
        const int cg = (f >> 4) * 32 + (f & 15), cu = cg + 16;
        const float g = c[cg] + (bias ? bias[cg] : 0.f), u = c[cu] + (bias ? bias[cu] : 0.f);
        ((T*)e.out_t)[(size_t)ra * e.ld_t + f] = from_f<T>(silu_f(g) * u);
      }
      return;
    default:
      break;
  }
  // EPI_QKV / EPI_KV: columns [0, n_q) query, [n_q, n_q + n_kv) key, then value.
  const int tok = e.row_tok[ra];
  const int seq = e.tok_seq[tok], pos = e.tok_pos[tok];
  const int dh = e.head_dim, half = dh >> 1;
  const int nq = e.n_q_cols, nkv = e.n_kv_cols;
  const long long base = e.cache.checked_base(e.layer0, seq, pos);
  T* kc = (T*)e.cache.k;
  T* vc = (T*)e.cache.v;
  // query and key pairs (RoPE rotate-half: feature i pairs with i + dh/2)
  const int n_pairs = (nq + nkv) / 2;
  for (int p = threadIdx.x; p < n_pairs; p += blockDim.x) {
    const int isk = p >= nq / 2;
    const int pp = isk ? p - nq / 2 : p;
    const int h = pp / half, i = pp % half;
    const int c1 = (isk ? nq : 0) + h * dh + i, c2 = c1 + half;
    float x1 = c[c1] + (bias ? bias[c1] : 0.f), x2 = c[c2] + (bias ? bias[c2] : 0.f);
    if (e.rope) {
      const float2 cs = e.rope_table[(size_t)pos * half + i];
      const float y1 = x1 * cs.x - x2 * cs.y, y2 = x2 * cs.x + x1 * cs.y;
      x1 = y1;
      x2 = y2;
    }
    if (!isk) {
      T* q = (T*)e.out_t + (size_t)ra * e.ld_t;
      q[h * dh + i] = from_f<T>(x1);
      q[h * dh + i + half] = from_f<T>(x2);
    } else if (base >= 0) {
      const size_t off = (size_t)base + h * e.cache.head_stride();
      kc[off + i] = from_f<T>(x1);
      kc[off + i + half] = from_f<T>(x2);
    }
  }
  if (base < 0) return;
  for (int n = threadIdx.x; n < nkv; n += blockDim.x) {
    const int cc = nq + nkv + n;
    const int h = n / dh, d = n % dh;
    vc[(size_t)base + h * e.cache.head_stride() + d] = from_f<T>(c[cc] + (bias ? bias[cc] : 0.f));
  }
}

void launch_gemm_simt(cudaStream_t st, int dt, const GemmProblem& p, int max_rows, float* scratch) {
  if (max_rows <= 0) return;
  dim3 grid(cdiv(p.N, 64), cdiv(max_rows, 64));
  if (dt == 1) {
    gemm_simt_kernel<bf16><<<grid, 256, 0, st>>>((const bf16*)p.A, p.lda, (const bf16*)p.B, p.ldb, p.rows, p.N, p.K,
                                                 scratch, p.N);
    epilogue_kernel<bf16><<<max_rows, 256, 0, st>>>(p.epi, scratch, p.N, p.rows, p.N);
  } else {
    gemm_simt_kernel<float><<<grid, 256, 0, st>>>((const float*)p.A, p.lda, (const float*)p.B, p.ldb, p.rows, p.N,
                                                  p.K, scratch, p.N);
    epilogue_kernel<float><<<max_rows, 256, 0, st>>>(p.epi, scratch, p.N, p.rows, p.N);
  }
}

}  // namespace adept

// Kernels of the HSM training step (Sec. 4.2; Sec. 5.1 "Training"; App. D): the Hidden State
// Mapper is trained with the base model frozen, by cross-entropy of its mapped state, read
// through the frozen final norm and LM head, against the next token, and AdamW.  Encoders
// (Sec. 4.3) train it by the cosine similarity of the mapped state to the original final
// state plus the frozen pooler + classifier's cross-entropy on the labelled [CLS] rows.
//
// The products (the four FC layers of Table S1, their input and weight gradients, the head
// and its input gradient) run on the library's GEMMs; these kernels are the elementwise and
// row-wise steps between them (GELU and its derivative, the softmax cross-entropy, the
// similarity and classifier rows, the RMSNorm / LayerNorm backward, the convolution
// backward), the deterministic column sums that give bias, gain and convolution gradients,
// operand transposes, and the AdamW update.
#define ADEPT_TU_ID 9
#include "common.cuh"
#include "hsm_train.h"

#include <algorithm>

namespace adept {

namespace {

// ---------------------------------------------------------------------------
// forward
// ---------------------------------------------------------------------------

template <typename T> __device__ __forceinline__ void store4(T* p, float a, float b, float c, float d);
template <> __device__ __forceinline__ void store4<float>(float* p, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
}
template <> __device__ __forceinline__ void store4<bf16>(bf16* p, float a, float b, float c, float d) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  uint2 u;
  u.x = *reinterpret_cast<unsigned*>(&lo);
  u.y = *reinterpret_cast<unsigned*>(&hi);
  *reinterpret_cast<uint2*>(p) = u;
}

// Softmax cross-entropy of one row of logits against its target (one CTA per row):
// lossr[r] = logsumexp(l) - l[target]; dl[r][v] = (softmax(l)_v - [v == target]) / n for
// v < V and 0 for the padding columns V..Vp-1.  A target outside [0, V) flags ERRW_TOKEN and
// leaves a zero loss and gradient for the row.  Rows are read as float4 groups (ldl and Vp
// multiples of 4; columns at or past V are masked), four groups in flight per thread; the
// second pass finds the row in L2 (512-thread CTAs, two per SM: one CTA's reductions overlap
// the other's loads, and ~300 rows in flight stay well inside L2 for vocabularies of ~50 K).
template <typename T>
__global__ void __launch_bounds__(512, 2) ht_ce_kernel(const float* __restrict__ logits, int ldl, int V, int Vp,
                                                     const int* __restrict__ target, float inv_n, float* lossr, T* dl,
                                                     unsigned* err) {
  PDL_ENTRY();
  __shared__ float red[32];
  __shared__ float rmax[32];
  const int r = blockIdx.x;
  const float4* l4 = reinterpret_cast<const float4*>(logits + (size_t)r * ldl);
  T* g = dl + (size_t)r * Vp;
  const int n4 = Vp >> 2;
  const int tg = target[r];
  if (tg < 0 || tg >= V) {
    if (threadIdx.x == 0) {
      atomicOr(err, ERRW_TOKEN);
      lossr[r] = 0.f;
    }
    for (int j = threadIdx.x; j < n4; j += blockDim.x) store4<T>(g + 4 * j, 0.f, 0.f, 0.f, 0.f);
    return;
  }
  // online (max, sum of exp) per thread, then across the block
  float mx = -INFINITY, s = 0.f;
  constexpr int U = 4;
  for (int j0 = threadIdx.x; j0 < n4; j0 += U * blockDim.x) {
    float4 x[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = j0 + u * blockDim.x;
      x[u] = j < n4 ? l4[j] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = j0 + u * blockDim.x;
      const int v = 4 * j;
      const float a0 = v < V ? x[u].x : -INFINITY, a1 = v + 1 < V ? x[u].y : -INFINITY;
      const float a2 = v + 2 < V ? x[u].z : -INFINITY, a3 = v + 3 < V ? x[u].w : -INFINITY;
      const float m4 = fmaxf(fmaxf(a0, a1), fmaxf(a2, a3));
      if (m4 == -INFINITY) continue;
      if (m4 > mx) {
        s *= expf(mx - m4);
        mx = m4;
      }
      s += expf(a0 - mx) + expf(a1 - mx) + expf(a2 - mx) + expf(a3 - mx);
    }
  }
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  float bm = warp_max(mx);
  if (lane == 0) rmax[w] = bm;
  __syncthreads();
  bm = -INFINITY;
  for (int i = 0; i < nw; ++i) bm = fmaxf(bm, rmax[i]);
  const float S = block_sum(mx == -INFINITY ? 0.f : s * expf(mx - bm), red);
  const float inv_s = 1.f / S;
  if (threadIdx.x == 0) lossr[r] = logf(S) + bm - reinterpret_cast<const float*>(l4)[tg];
  for (int j = threadIdx.x; j < n4; j += blockDim.x) {
    const float4 x = l4[j];
    const int v = 4 * j;
    const float xv[4] = {x.x, x.y, x.z, x.w};
    float d[4];
#pragma unroll
    for (int q = 0; q < 4; ++q)
      d[q] = v + q < V ? (expf(xv[q] - bm) * inv_s - (v + q == tg ? 1.f : 0.f)) * inv_n : 0.f;
    store4<T>(g + v, d[0], d[1], d[2], d[3]);
  }
}

// loss = scale * sum_r lossr[r] (+ scale_b * sum_r lossb[r]) in a fixed order (one CTA).
__global__ void ht_loss_kernel(const float* lossr, int n, float scale, const float* lossb, int nb, float scale_b,
                               float* loss) {
  PDL_ENTRY();
  __shared__ float red[32];
  float s = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += lossr[i];
  s = block_sum(s, red);
  float sb = 0.f;
  for (int i = threadIdx.x; i < nb; i += blockDim.x) sb += lossb[i];
  sb = block_sum(sb, red);
  if (threadIdx.x == 0) *loss = s * scale + (nb ? sb * scale_b : 0.f);
}

// Similarity loss rows of the encoder step (Sec. 4.3; one CTA per row): with s = s~_r and
// t = s_N,r, lossr[r] = 1 - cos, cos = s.t / (|s| |t|), and the row's gradient
//   dxh[r] = -inv_n (t / (|s| |t|) - cos s / |s|^2)
// (cos = 0 and no gradient where |s| |t| = 0).
__global__ void ht_cos_kernel(const float* __restrict__ st, const float* __restrict__ tg, int D, float inv_n,
                              float* lossr, float* dxh) {
  PDL_ENTRY();
  __shared__ float red[32];
  const size_t o = (size_t)blockIdx.x * D;
  float a = 0.f, ss = 0.f, tt = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float s = st[o + d], t = tg[o + d];
    a += s * t;
    ss += s * s;
    tt += t * t;
  }
  a = block_sum(a, red);
  ss = block_sum(ss, red);
  tt = block_sum(tt, red);
  float cs = 0.f, ct = 0.f, cosv = 0.f;
  if (ss > 0.f && tt > 0.f) {
    const float den = sqrtf(ss) * sqrtf(tt);
    cosv = a / den;
    ct = -inv_n / den;
    cs = inv_n * cosv / ss;
  }
  for (int d = threadIdx.x; d < D; d += blockDim.x) dxh[o + d] = ct * tg[o + d] + cs * st[o + d];
  if (threadIdx.x == 0) lossr[blockIdx.x] = 1.f - cosv;
}

template <typename T> __device__ __forceinline__ float round_to(float x) { return to_f<T>(from_f<T>(x)); }

// Task loss of the encoder step (Sec. 4.3) on the labelled rows (one CTA per row): pooled =
// tanh(zp) (zp: the pooler's pre-activation, bias included), logits z_c = round(pooled) . Wc[c]
// + bc[c], lossc[r] = logsumexp(z) - z[label]; with dz_c = scale (softmax(z)_c - [c = label])
// rounded like a GEMM input, dpt[r][d] = (sum_c dz_c Wc[c][d]) (1 - pooled[d]^2), the gradient
// into the pooler's pre-activation (T, the next product's input).  A label outside [0, C)
// flags ERRW_LABEL and leaves a zero loss and gradient for the row.
template <typename T>
__global__ void ht_cls_kernel(const float* __restrict__ zp, int D, const T* __restrict__ wc,
                              const float* __restrict__ bc, int C, const int* __restrict__ label, float scale,
                              float* lossc, T* dpt, unsigned* err) {
  PDL_ENTRY();
  __shared__ float red[32];
  __shared__ float dz[HT_MAX_CLASSES];
  const size_t o = (size_t)blockIdx.x * D;
  const int y = label[blockIdx.x];
  if (y < 0 || y >= C) {
    if (threadIdx.x == 0) {
      atomicOr(err, ERRW_LABEL);
      lossc[blockIdx.x] = 0.f;
    }
    for (int d = threadIdx.x; d < D; d += blockDim.x) dpt[o + d] = from_f<T>(0.f);
    return;
  }
  for (int c = 0; c < C; ++c) {
    float s = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s += round_to<T>(tanhf(zp[o + d])) * to_f(wc[(size_t)c * D + d]);
    s = block_sum(s, red);
    if (threadIdx.x == 0) dz[c] = s + bc[c];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float mx = -INFINITY;
    for (int c = 0; c < C; ++c) mx = fmaxf(mx, dz[c]);
    float S = 0.f;
    for (int c = 0; c < C; ++c) S += expf(dz[c] - mx);
    lossc[blockIdx.x] = logf(S) + mx - dz[y];
    for (int c = 0; c < C; ++c) dz[c] = round_to<T>(scale * (expf(dz[c] - mx) / S - (c == y ? 1.f : 0.f)));
  }
  __syncthreads();
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    float g = 0.f;
    for (int c = 0; c < C; ++c) g += dz[c] * to_f(wc[(size_t)c * D + d]);
    const float p = tanhf(zp[o + d]);
    dpt[o + d] = from_f<T>(g * (1.f - p * p));
  }
}

// ---------------------------------------------------------------------------
// backward
// ---------------------------------------------------------------------------

// Through the frozen head's standardisation and the HSM's last block (one CTA per row).
// st = s~ = RMSNorm_g2(h5) + c0; xh = standardise(st) (LayerNorm without affine for mode LN,
// RMS scaling for mode RMS; the head's gain and bias are folded into its weights; mode COPY,
// the encoder's post-LN final state, reads s~ itself: dst = dxh).
//   dst = rstd (dxh - mean(dxh) - xh mean(dxh xh))          (LN; RMS drops mean(dxh))
//   dc0 = dst;  dr = dst g2;  dh5 = r2 (dr - rh mean(dr rh)),  rh = h5 r2
// Writes dc0 (fp32), dh5 (fp32 and T) and r2 (for the g2 column sum).
// dxh arrives as nsplit partial sums (K-split parts of the head's input-gradient product),
// split_stride floats apart.
template <typename T>
__global__ void ht_out_bwd_kernel(const float* __restrict__ dxh, int nsplit, size_t split_stride,
                                  const float* __restrict__ st, const float* __restrict__ h5, int D,
                                  const float* __restrict__ g2, float eps, int mode, float norm_eps, float* dc0,
                                  float* dh5f, T* dh5t, float* r2_out) {
  PDL_ENTRY();
  __shared__ float red[32];
  const size_t o = (size_t)blockIdx.x * D;
  const float *f = st + o, *h = h5 + o;
  auto X = [&](int d) {
    float v = dxh[o + d];
    for (int s = 1; s < nsplit; ++s) v += dxh[s * split_stride + o + d];
    return v;
  };
  float q2 = 0.f;
  if (mode == NORM_COPY) {
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      dc0[o + d] = X(d);
      q2 += h[d] * h[d];
    }
  } else {
    float mu = 0.f;
    if (mode == NORM_LN) {
      float s = 0.f;
      for (int d = threadIdx.x; d < D; d += blockDim.x) s += f[d];
      mu = block_sum(s, red) / D;
    }
    float s2 = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      const float c = f[d] - mu;
      s2 += c * c;
    }
    const float rs = rsqrtf(block_sum(s2, red) / D + norm_eps);
    float sa = 0.f, sb = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      const float xd = X(d);
      sa += xd;
      sb += xd * (f[d] - mu) * rs;
    }
    const float ma = mode == NORM_LN ? block_sum(sa, red) / D : 0.f;
    const float mb = block_sum(sb, red) / D;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      const float v = rs * (X(d) - ma - (f[d] - mu) * rs * mb);
      dc0[o + d] = v;
      q2 += h[d] * h[d];
    }
  }
  const float r2 = rsqrtf(block_sum(q2, red) / D + eps);
  float sc = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) sc += dc0[o + d] * g2[d] * h[d] * r2;
  const float mc = block_sum(sc, red) / D;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float v = r2 * (dc0[o + d] * g2[d] - h[d] * r2 * mc);
    dh5f[o + d] = v;
    dh5t[o + d] = from_f<T>(v);
  }
  if (threadIdx.x == 0) r2_out[blockIdx.x] = r2;
}

// Through h4 = RMSNorm_g1(h3) + h1 (one CTA per row): dh3 = r1 (dh4 g1 - rh mean(dh4 g1 rh)),
// rh = h3 r1.  The h1 branch's gradient is dh4 itself (kept in place by the caller).
template <typename T>
__global__ void ht_mid_bwd_kernel(const float* __restrict__ dh4, const float* __restrict__ h3, int m1,
                                  const float* __restrict__ g1, float eps, float* dh3f, T* dh3t, float* r1_out) {
  PDL_ENTRY();
  __shared__ float red[32];
  const size_t o = (size_t)blockIdx.x * m1;
  const float *x = dh4 + o, *h = h3 + o;
  float q2 = 0.f;
  for (int d = threadIdx.x; d < m1; d += blockDim.x) q2 += h[d] * h[d];
  const float r1 = rsqrtf(block_sum(q2, red) / m1 + eps);
  float sc = 0.f;
  for (int d = threadIdx.x; d < m1; d += blockDim.x) sc += x[d] * g1[d] * h[d] * r1;
  const float mc = block_sum(sc, red) / m1;
  for (int d = threadIdx.x; d < m1; d += blockDim.x) {
    const float v = r1 * (x[d] * g1[d] - h[d] * r1 * mc);
    dh3f[o + d] = v;
    dh3t[o + d] = from_f<T>(v);
  }
  if (threadIdx.x == 0) r1_out[blockIdx.x] = r1;
}

// Through the convolution and the input RMSNorms (one CTA per row).  With Xn_a = xh_a g0,
// xh_a = u_a rstd_a (u: s_i, s_{i-1}, I) and c0[d] = b + sum_{a,u} w[a][u] Xn_a[d + u - 1]:
//   dXn_a[j] = sum_u w[a][u] dc0[j - u + 1]       -> pg0[j] = sum_a dXn_a[j] xh_a[j]
//   dw[a][u] = sum_d dc0[d] Xn_a[d + u - 1],  db = sum_d dc0[d]   -> cw[row][10]
// (The inputs are data: no gradient flows into them.)
__global__ void ht_prep_bwd_kernel(const float* __restrict__ hs, const float* __restrict__ hp,
                                   const float* __restrict__ hI, const float* __restrict__ dc0, int D,
                                   const float* __restrict__ g0, const float* __restrict__ conv, float eps,
                                   float* pg0, float* cw) {
  PDL_ENTRY();
  __shared__ float red[32];
  const size_t o = (size_t)blockIdx.x * D;
  const float* x[3] = {hs + o, hp + o, hI + o};
  const float* dc = dc0 + o;
  float sc[3];
#pragma unroll
  for (int a = 0; a < 3; ++a) {
    float s2 = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s2 += x[a][d] * x[a][d];
    sc[a] = rsqrtf(block_sum(s2, red) / D + eps);
  }
  float acc[10];
#pragma unroll
  for (int i = 0; i < 10; ++i) acc[i] = 0.f;
  for (int j = threadIdx.x; j < D; j += blockDim.x) {
    float p = 0.f;
    const float dcj = dc[j];
#pragma unroll
    for (int a = 0; a < 3; ++a) {
      float dx = 0.f;
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int t = j - u + 1;   // output column fed by Xn_a[j] through tap u
        if (t >= 0 && t < D) dx += conv[a * 3 + u] * dc[t];
        const int s = j + u - 1;   // input column tap u reads for output column j
        if (s >= 0 && s < D) acc[a * 3 + u] += dcj * x[a][s] * sc[a] * g0[s];
      }
      p += dx * x[a][j] * sc[a];
    }
    acc[9] += dcj;
    pg0[o + j] = p;
  }
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const float t = block_sum(acc[i], red);
    if (threadIdx.x == 0) cw[(size_t)blockIdx.x * 10 + i] = t;
  }
}

// ---------------------------------------------------------------------------
// column sums (deterministic: fixed row chunks, then a fixed-order sum of the chunks)
// ---------------------------------------------------------------------------

__global__ void ht_colsum_kernel(ColJobs J, float* part, int ctot) {
  PDL_ENTRY();
  int j = 0;
  while (j + 1 < J.nj && (int)blockIdx.x >= J.cb[j + 1]) ++j;
  const ColJob& q = J.j[j];
  const int c = (blockIdx.x - J.cb[j]) * blockDim.x + threadIdx.x;
  if (c >= q.C) return;
  const int r0 = blockIdx.y * J.rows_per, r1 = min(J.n, r0 + J.rows_per);
  float s = 0.f;
  for (int r = r0; r < r1; ++r) {
    float v = q.A[(size_t)r * q.C + c];
    if (q.B) v *= q.B[(size_t)r * q.C + c];
    if (q.rs) v *= q.rs[r];
    s += v;
  }
  part[(size_t)blockIdx.y * ctot + J.pc[j] + c] = s;
}

// Sum of the chunk partials per column: a block of 32 columns x 8 warps, warp w adding the
// chunks w, w + 8, ..., then the 8 warp sums in a fixed order.
__global__ void ht_colsum_finish_kernel(ColJobs J, const float* part, int ctot, int chunks) {
  PDL_ENTRY();
  __shared__ float acc[8][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int i = blockIdx.x * 32 + tx;
  float s = 0.f;
  if (i < ctot)
    for (int y = ty; y < chunks; y += 8) s += part[(size_t)y * ctot + i];
  acc[ty][tx] = s;
  __syncthreads();
  if (ty != 0 || i >= ctot) return;
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) t += acc[w][tx];
  int j = 0;
  while (j + 1 < J.nj && i >= J.pc[j + 1]) ++j;
  J.j[j].out[i - J.pc[j]] = t;
}

// Elementwise GELU steps that also write their result transposed (32 x 32 tiles through shared
// memory), for the weight-gradient products that read it as their K-major operand:
//   BWD = 0 (forward):  h = GELU_erf(z)            -> hf (optional, fp32), ht [n][C], hT [C][ldT]
//   BWD = 1 (backward): dz = dh GELU_erf'(z)      -> dh (in place, fp32), ht [n][C], hT [C][ldT]
// Rows n..ldT-1 of the tile grid only write zeros into hT's padding columns.
// BWD = 1 also writes the tile's column sums over its 32 rows into part[blockIdx.y][C] (the
// chunk partials of the bias gradient, HT_COLSUM_ROWS = 32).
template <typename T, int BWD>
__global__ void ht_gelu_tile_kernel(const float* __restrict__ z, float* hf, int n, int C, T* ht, T* hT, int ldT,
                                    float* part) {
  PDL_ENTRY();
  __shared__ float tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int r = r0 + i, c = c0 + tx;
    float v = 0.f;
    if (r < n && c < C) {
      const size_t e = (size_t)r * C + c;
      const float x = z[e];
      if (BWD) {
        const float gp =
            0.5f * (1.f + erff(x * 0.70710678118654752f)) + x * 0.39894228040143268f * expf(-0.5f * x * x);
        v = hf[e] * gp;
        hf[e] = v;
      } else {
        v = gelu_erf_f(x);
        if (hf) hf[e] = v;
      }
      ht[e] = from_f<T>(v);
    }
    tile[i][tx] = v;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int c = c0 + i, r = r0 + tx;
    if (c < C && r < ldT) hT[(size_t)c * ldT + r] = from_f<T>(tile[tx][i]);
  }
  if (BWD && ty == 0 && c0 + tx < C) {
    float cs = 0.f;
    for (int i = 0; i < 32; ++i) cs += tile[i][tx];
    part[(size_t)blockIdx.y * C + c0 + tx] = cs;
  }
}

// ---------------------------------------------------------------------------
// transposes and the optimiser
// ---------------------------------------------------------------------------

// dst[c][r] = src[r][c] for r < n, 0 for n <= r < ldT (32 x 32 tiles through shared memory).
template <typename T>
__global__ void ht_transpose_kernel(const T* __restrict__ src, int n, int C, T* dst, int ldT) {
  PDL_ENTRY();
  __shared__ float tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int r = r0 + i, c = c0 + tx;
    tile[i][tx] = (r < n && c < C) ? to_f(src[(size_t)r * C + c]) : 0.f;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int c = c0 + i, r = r0 + tx;
    if (c < C && r < ldT) dst[(size_t)c * ldT + r] = from_f<T>(tile[tx][i]);
  }
}

// AdamW (decoupled weight decay, bias-corrected moments) over every parameter segment in
// 32 x 32 tiles; each updated value is also written to the segment's fp32 copy, its T copy
// and (through shared memory) its transposed T copy, whichever are given.
template <typename T>
__global__ void ht_adamw_kernel(AdamArgs A) {
  PDL_ENTRY();
  __shared__ float tile[32][33];
  int s = 0;
  while (s + 1 < A.nseg && (int)blockIdx.x >= A.seg[s + 1].tile0) ++s;
  const AdamSeg& g = A.seg[s];
  const int t = blockIdx.x - g.tile0;
  const int tr = t / g.tiles_x, tc = t % g.tiles_x;
  const int r0 = tr * 32, c0 = tc * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int r = r0 + i, c = c0 + tx;
    if (r >= g.rows || c >= g.cols) continue;
    const size_t e = (size_t)r * g.cols + c;
    const size_t k = (size_t)g.off + e;
    const float gr = A.grad[k];
    const float m = A.b1 * A.m[k] + (1.f - A.b1) * gr;
    const float v = A.b2 * A.v[k] + (1.f - A.b2) * gr * gr;
    float th = A.theta[k];
    th = th - A.lr * A.wd * th - A.lr * (m * A.ibc1) / (sqrtf(v * A.ibc2) + A.eps);
    A.m[k] = m;
    A.v[k] = v;
    A.theta[k] = th;
    if (g.wf) g.wf[e] = th;
    if (g.wt) ((T*)g.wt)[e] = from_f<T>(th);
    tile[i][tx] = th;
  }
  if (!g.wT) return;
  __syncthreads();
  for (int i = ty; i < 32; i += blockDim.x >> 5) {
    const int c = c0 + i, r = r0 + tx;
    if (c < g.cols && r < g.rows) ((T*)g.wT)[(size_t)c * g.rows + r] = from_f<T>(tile[tx][i]);
  }
}

}  // namespace

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------

void ht_launch_ce(cudaStream_t st, int dt, const float* logits, int ldl, int n, int V, int Vp, const int* target,
                  float* lossr, void* dl, float* loss, unsigned* err) {
  const float inv_n = 1.f / (float)n;
  if (dt == 1) launch_k(ht_ce_kernel<bf16>, n, 512, 0, st, logits, ldl, V, Vp, target, inv_n, lossr, (bf16*)dl, err);
  else launch_k(ht_ce_kernel<float>, n, 512, 0, st, logits, ldl, V, Vp, target, inv_n, lossr, (float*)dl, err);
  if (loss) launch_k(ht_loss_kernel, 1, 1024, 0, st, (const float*)lossr, n, inv_n, (const float*)nullptr, 0, 0.f, loss);
}

void ht_launch_cos(cudaStream_t st, const float* stv, const float* tgt, int n, int D, float* lossr, float* dxh) {
  launch_k(ht_cos_kernel, n, 256, 0, st, stv, tgt, D, 1.f / (float)n, lossr, dxh);
}

void ht_launch_cls(cudaStream_t st, int dt, const float* zp, int n_cls, int D, const void* wc, const float* bc, int C,
                   const int* label, float scale, float* lossc, void* dpt, unsigned* err) {
  if (dt == 1)
    launch_k(ht_cls_kernel<bf16>, n_cls, 256, 0, st, zp, D, (const bf16*)wc, bc, C, label, scale, lossc, (bf16*)dpt,
             err);
  else
    launch_k(ht_cls_kernel<float>, n_cls, 256, 0, st, zp, D, (const float*)wc, bc, C, label, scale, lossc,
             (float*)dpt, err);
}

void ht_launch_loss(cudaStream_t st, const float* la, int na, float sa, const float* lb, int nb, float sb,
                    float* loss) {
  launch_k(ht_loss_kernel, 1, 1024, 0, st, la, na, sa, lb, nb, sb, loss);
}

void ht_launch_out_bwd(cudaStream_t st, int dt, const float* dxh, int nsplit, size_t split_stride, const float* stv,
                       const float* h5, int n, int D, const float* g2, float eps, int mode, float norm_eps, float* dc0,
                       float* dh5f, void* dh5t, float* r2) {
  if (dt == 1)
    launch_k(ht_out_bwd_kernel<bf16>, n, 256, 0, st, dxh, nsplit, split_stride, stv, h5, D, g2, eps, mode, norm_eps,
             dc0, dh5f, (bf16*)dh5t, r2);
  else
    launch_k(ht_out_bwd_kernel<float>, n, 256, 0, st, dxh, nsplit, split_stride, stv, h5, D, g2, eps, mode, norm_eps,
             dc0, dh5f, (float*)dh5t, r2);
}

void ht_launch_mid_bwd(cudaStream_t st, int dt, const float* dh4, const float* h3, int n, int m1, const float* g1,
                       float eps, float* dh3f, void* dh3t, float* r1) {
  if (dt == 1) launch_k(ht_mid_bwd_kernel<bf16>, n, 256, 0, st, dh4, h3, m1, g1, eps, dh3f, (bf16*)dh3t, r1);
  else launch_k(ht_mid_bwd_kernel<float>, n, 256, 0, st, dh4, h3, m1, g1, eps, dh3f, (float*)dh3t, r1);
}

void ht_launch_gelu_tile(cudaStream_t st, int dt, int bwd, const float* z, float* hf, int n, int C, void* ht, void* hT,
                         int ldT, float* part) {
  const dim3 grid((C + 31) / 32, (ldT + 31) / 32);
  if (dt == 1) {
    if (bwd) launch_k(ht_gelu_tile_kernel<bf16, 1>, grid, 256, 0, st, z, hf, n, C, (bf16*)ht, (bf16*)hT, ldT, part);
    else launch_k(ht_gelu_tile_kernel<bf16, 0>, grid, 256, 0, st, z, hf, n, C, (bf16*)ht, (bf16*)hT, ldT, part);
  } else {
    if (bwd) launch_k(ht_gelu_tile_kernel<float, 1>, grid, 256, 0, st, z, hf, n, C, (float*)ht, (float*)hT, ldT, part);
    else launch_k(ht_gelu_tile_kernel<float, 0>, grid, 256, 0, st, z, hf, n, C, (float*)ht, (float*)hT, ldT, part);
  }
}

void ht_launch_prep_bwd(cudaStream_t st, const float* hs, const float* hp, const float* hI, const float* dc0, int n,
                        int D, const float* g0, const float* conv, float eps, float* pg0, float* cw) {
  launch_k(ht_prep_bwd_kernel, n, 256, 0, st, hs, hp, hI, dc0, D, g0, conv, eps, pg0, cw);
}

int ht_colsum_chunks(int n) { return (n + HT_COLSUM_ROWS - 1) / HT_COLSUM_ROWS; }

static void colsum_layout(ColJobs& J, int* nb, int* ctot) {
  *ctot = 0;
  *nb = 0;
  for (int j = 0; j < J.nj; ++j) {
    J.cb[j] = *nb;
    J.pc[j] = *ctot;
    *nb += (J.j[j].C + 255) / 256;
    *ctot += J.j[j].C;
  }
  J.cb[J.nj] = *nb;
  J.pc[J.nj] = *ctot;
  J.rows_per = HT_COLSUM_ROWS;
}

int ht_launch_colsum(cudaStream_t st, ColJobs J, float* part) {
  int ctot = 0, nb = 0;
  colsum_layout(J, &nb, &ctot);
  const int chunks = ht_colsum_chunks(J.n);
  launch_k(ht_colsum_kernel, dim3(nb, chunks), 256, 0, st, J, part, ctot);
  launch_k(ht_colsum_finish_kernel, (ctot + 31) / 32, 256, 0, st, J, (const float*)part, ctot, chunks);
  return 2;
}

int ht_launch_colsum_finish(cudaStream_t st, ColJobs J, const float* part) {
  int ctot = 0, nb = 0;
  colsum_layout(J, &nb, &ctot);
  launch_k(ht_colsum_finish_kernel, (ctot + 31) / 32, 256, 0, st, J, part, ctot, ht_colsum_chunks(J.n));
  return 1;
}

void ht_launch_transpose(cudaStream_t st, int dt, const void* src, int n, int C, void* dst, int ldT) {
  const dim3 grid((C + 31) / 32, (ldT + 31) / 32);
  if (dt == 1) launch_k(ht_transpose_kernel<bf16>, grid, 256, 0, st, (const bf16*)src, n, C, (bf16*)dst, ldT);
  else launch_k(ht_transpose_kernel<float>, grid, 256, 0, st, (const float*)src, n, C, (float*)dst, ldT);
}

void ht_launch_adamw(cudaStream_t st, int dt, AdamArgs A) {
  int tiles = 0;
  for (int s = 0; s < A.nseg; ++s) {
    A.seg[s].tiles_x = (A.seg[s].cols + 31) / 32;
    A.seg[s].tile0 = tiles;
    tiles += ((A.seg[s].rows + 31) / 32) * A.seg[s].tiles_x;
  }
  if (dt == 1) launch_k(ht_adamw_kernel<bf16>, tiles, 256, 0, st, A);
  else launch_k(ht_adamw_kernel<float>, tiles, 256, 0, st, A);
}

ADEPT_KTRACE_ATTACH(hsm_train)

}  // namespace adept

// Attention of the active query rows over the paged KV cache of one layer.  The keys
// of a sequence at layer i are every cached position of that layer -- computed by the
// token itself if it was active at i, or filled from its mapped state s~_N if it
// exited earlier -- so attention needs no knowledge of exits.
#define ADEPT_TU_ID 1
#include "common.cuh"
#include "kernels.h"
#include "attention_tc.h"

#include <algorithm>

namespace adept {

// One warp per (query row, head); lanes own keys for the scores and head dimensions
// for the value sum; online softmax over blocks of 32 keys.
template <typename T, int DH>
__global__ void __launch_bounds__(256) attn_warp_kernel(const T* __restrict__ q, int ld_q, T* __restrict__ out,
                                                        int ld_out, DevRange rows, const int* row_tok,
                                                        const int* tok_seq, const int* tok_pos, const int* seq_len,
                                                        KVCacheView cache, int layer0, int n_heads, int causal,
                                                        float scale) {
  PDL_ENTRY();
  __shared__ float qs[8][DH];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * 8 + warp;
  const int rb = rows.b(), M = rows.e() - rb;
  const int r = gw / n_heads, h = gw % n_heads;
  if (r >= M) return;
  const int ra = rb + r;
  const int tok = row_tok[ra];
  const int seq = tok_seq[tok], pos = tok_pos[tok];
  const int kvh = h / (n_heads / cache.n_kv_heads);
  for (int d = lane; d < DH; d += 32) qs[warp][d] = to_f(q[(size_t)ra * ld_q + h * DH + d]) * scale;
  __syncwarp();
  const int nk = causal ? pos + 1 : seq_len[seq];
  const T* K = (const T*)cache.k;
  const T* V = (const T*)cache.v;
  constexpr int PER = DH / 32;
  float acc[PER];
#pragma unroll
  for (int j = 0; j < PER; ++j) acc[j] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int kb = 0; kb < nk; kb += 32) {
    const int key = kb + lane;
    float s = -INFINITY;
    if (key < nk) {
      const T* kr = K + cache.offset(layer0, seq, key, kvh);
      float a = 0.f;
#pragma unroll 8
      for (int d = 0; d < DH; ++d) a = fmaf(qs[warp][d], to_f(kr[d]), a);
      s = a;
    }
    const float mn = fmaxf(m, warp_max(s));
    const float p = key < nk ? expf(s - mn) : 0.f;
    const float corr = (m == -INFINITY) ? 0.f : expf(m - mn);
    l = l * corr + warp_sum(p);
#pragma unroll
    for (int j = 0; j < PER; ++j) acc[j] *= corr;
    const int nb = min(32, nk - kb);
    for (int kk = 0; kk < nb; ++kk) {
      const float pk = __shfl_sync(0xffffffffu, p, kk);
      const T* vr = V + cache.offset(layer0, seq, kb + kk, kvh);
#pragma unroll
      for (int j = 0; j < PER; ++j) acc[j] = fmaf(pk, to_f(vr[lane + 32 * j]), acc[j]);
    }
    m = mn;
  }
  const float inv = 1.f / l;
#pragma unroll
  for (int j = 0; j < PER; ++j) out[(size_t)ra * ld_out + h * DH + lane + 32 * j] = from_f<T>(acc[j] * inv);
}

// ---------------------------------------------------------------------------
// Prompt-pass attention, bf16 tensor cores (mma.sync m16n8k16): a CTA takes 64
// consecutive active query rows of one head.  Active rows are sorted by (sequence,
// position), so the tile splits into runs of one sequence; each run streams its keys
// [0, last position] (causal) or [0, length) from the paged cache in blocks of 64,
// with an online softmax (exp2 domain) per query row.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void ldsm_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3, const void* p) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3, const void* p) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(a), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// x = hi + lo with hi = bf16(x) and lo = bf16(x - hi), for a pair of values.
__device__ __forceinline__ void split_bf16(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
  const float2 hf = __bfloat1622float2(h);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = pack_bf16(x0 - hf.x, x1 - hf.y);
}

template <int DH>
__global__ void __launch_bounds__(128) attn_prefill_mma_kernel(const bf16* __restrict__ q, int ld_q,
                                                               bf16* __restrict__ out, int ld_out, DevRange rows,
                                                               const int* row_tok, const int* tok_seq,
                                                               const int* tok_pos, const int* seq_len,
                                                               KVCacheView cache, int layer0, int n_heads, int causal,
                                                               float scale_log2, const int* key_exit, int kp_len) {
  PDL_ENTRY();
  constexpr int LDS = DH + 8;  // padded rows: conflict-free ldmatrix
  constexpr int NB = DH / 8;   // 8-column blocks of the output
  extern __shared__ __align__(16) uint8_t attn_smem[];
  bf16* sQ = reinterpret_cast<bf16*>(attn_smem);
  bf16* sK = sQ + 64 * LDS;
  bf16* sV = sK + 64 * LDS;
  __shared__ int s_seq[64], s_pos[64];
  __shared__ int s_kv[64];   // key of the tile present (in range; with key_exit: still active)

  const int h = blockIdx.y;
  const int kvh = h / (n_heads / cache.n_kv_heads);
  const int r0 = rows.b() + blockIdx.x * 64;
  const int rend = rows.e();
  if (r0 >= rend) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t4 = lane & 3;
  if (tid < 64) {
    const int r = r0 + tid;
    if (r < rend) {
      const int tok = row_tok[r];
      s_seq[tid] = tok_seq[tok];
      s_pos[tid] = tok_pos[tok];
    } else {
      s_seq[tid] = -1;
      s_pos[tid] = -1;
    }
  }
  // Q tile (rows past the range are zero)
  for (int c = tid; c < 64 * (DH / 8); c += 128) {
    const int rr = c / (DH / 8), cc = (c % (DH / 8)) * 8;
    bf16* dst = sQ + rr * LDS + cc;
    if (r0 + rr < rend) cp_async16(dst, q + (size_t)(r0 + rr) * ld_q + h * DH + cc);
    else *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
  }
  cp_async_wait_all();
  __syncthreads();
  const bf16* Kp = (const bf16*)cache.k;
  const bf16* Vp = (const bf16*)cache.v;

  int a = 0;
  while (a < 64 && s_seq[a] >= 0) {
    const int sq = s_seq[a];
    int b = a;
    while (b < 64 && s_seq[b] == sq) ++b;
    const int kend = causal ? s_pos[b - 1] + 1 : seq_len[sq];
    // this warp's two rows per thread (tile rows 16 warp + g, + 8)
    const int ra_ = warp * 16 + g, rb_ = ra_ + 8;
    const bool va = ra_ >= a && ra_ < b, vb = rb_ >= a && rb_ < b;
    const int pa = va ? s_pos[ra_] : -1, pb = vb ? s_pos[rb_] : -1;
    const bool warp_active = (warp * 16 < b) && (warp * 16 + 16 > a);
    // Q fragments of this warp (16 rows x DH)
    uint32_t qf[DH / 16][4];
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
      const int mi = lane >> 3;
      const int row = warp * 16 + (mi & 1) * 8 + (lane & 7);
      const int col = kk * 16 + (mi >> 1) * 8;
      ldsm_x4(qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], sQ + row * LDS + col);
    }
    float o[NB][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) o[nb][0] = o[nb][1] = o[nb][2] = o[nb][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    for (int kb = 0; kb < kend; kb += 64) {
      __syncthreads();  // previous K/V tile fully consumed
      for (int c = tid; c < 64 * (DH / 8); c += 128) {
        const int j = c / (DH / 8), cc = (c % (DH / 8)) * 8;
        const int p = kb + j;
        bf16* dk = sK + j * LDS + cc;
        bf16* dv = sV + j * LDS + cc;
        // "stop entirely": a token that left before this layer has no K/V here
        const bool present = p < kend && (!key_exit || key_exit[sq * kp_len + p] > layer0);
        if (cc == 0) s_kv[j] = present;
        if (present) {
          const size_t off = cache.offset(layer0, sq, p, kvh) + cc;
          cp_async16(dk, Kp + off);
          cp_async16(dv, Vp + off);
        } else {
          *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
          *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
        }
      }
      cp_async_wait_all();
      __syncthreads();
      if (!warp_active) continue;
      // S = Q K^T for 64 keys (8 blocks of 8)
      float s[8][4];
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) s[nb][0] = s[nb][1] = s[nb][2] = s[nb][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {  // pairs of key blocks (16 keys)
          const int mi = lane >> 3;
          const int key = np * 16 + (mi >> 1) * 8 + (lane & 7);
          const int col = kk * 16 + (mi & 1) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(b0, b1, b2, b3, sK + key * LDS + col);
          mma_bf16_16816(s[2 * np], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b0, b1);
          mma_bf16_16816(s[2 * np + 1], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b2, b3);
        }
      }
      // mask and online softmax (two rows per thread)
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = kb + nb * 8 + 2 * t4 + e;
          const bool kp = s_kv[nb * 8 + 2 * t4 + e];
          const bool ka = va && kp && (!causal || key <= pa);
          const bool kb_ = vb && kp && (!causal || key <= pb);
          s[nb][e] = ka ? s[nb][e] * scale_log2 : -INFINITY;
          s[nb][2 + e] = kb_ ? s[nb][2 + e] * scale_log2 : -INFINITY;
          mx0 = fmaxf(mx0, s[nb][e]);
          mx1 = fmaxf(mx1, s[nb][2 + e]);
        }
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float c0 = (mn0 == -INFINITY) ? 1.f : exp2f(m0 - mn0);
      const float c1 = (mn1 == -INFINITY) ? 1.f : exp2f(m1 - mn1);
      float sum0 = 0.f, sum1 = 0.f;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const float p0 = (s[nb][e] == -INFINITY) ? 0.f : exp2f(s[nb][e] - mn0);
          const float p1 = (s[nb][2 + e] == -INFINITY) ? 0.f : exp2f(s[nb][2 + e] - mn1);
          s[nb][e] = p0;
          s[nb][2 + e] = p1;
          sum0 += p0;
          sum1 += p1;
        }
      }
      sum0 += __shfl_xor_sync(0xffffffffu, sum0, 1);
      sum0 += __shfl_xor_sync(0xffffffffu, sum0, 2);
      sum1 += __shfl_xor_sync(0xffffffffu, sum1, 1);
      sum1 += __shfl_xor_sync(0xffffffffu, sum1, 2);
      l0 = l0 * c0 + sum0;
      l1 = l1 * c1 + sum1;
      m0 = mn0;
      m1 = mn1;
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        o[nb][0] *= c0;
        o[nb][1] *= c0;
        o[nb][2] *= c1;
        o[nb][3] *= c1;
      }
      // O += P V, with P = hi + lo (two bf16 terms) so the probabilities keep ~16 bits
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) {  // 16 keys per step
        uint32_t ah[4], al[4];
        split_bf16(s[2 * kc][0], s[2 * kc][1], ah[0], al[0]);
        split_bf16(s[2 * kc][2], s[2 * kc][3], ah[1], al[1]);
        split_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1], ah[2], al[2]);
        split_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3], ah[3], al[3]);
#pragma unroll
        for (int np = 0; np < NB / 2; ++np) {  // pairs of 8-column output blocks
          const int mi = lane >> 3;
          const int key = kc * 16 + (mi & 1) * 8 + (lane & 7);
          const int col = np * 16 + (mi >> 1) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(b0, b1, b2, b3, sV + key * LDS + col);
          mma_bf16_16816(o[2 * np], ah[0], ah[1], ah[2], ah[3], b0, b1);
          mma_bf16_16816(o[2 * np + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
          mma_bf16_16816(o[2 * np], al[0], al[1], al[2], al[3], b0, b1);
          mma_bf16_16816(o[2 * np + 1], al[0], al[1], al[2], al[3], b2, b3);
        }
      }
    }
    // normalise and write this warp's rows of the run
    const float i0 = l0 > 0.f ? 1.f / l0 : 0.f, i1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      const int col = h * DH + nb * 8 + 2 * t4;
      if (va) *reinterpret_cast<uint32_t*>(out + (size_t)(r0 + ra_) * ld_out + col) = pack_bf16(o[nb][0] * i0, o[nb][1] * i0);
      if (vb) *reinterpret_cast<uint32_t*>(out + (size_t)(r0 + rb_) * ld_out + col) = pack_bf16(o[nb][2] * i1, o[nb][3] * i1);
    }
    a = b;
  }
}

// ---------------------------------------------------------------------------
// Generation-step attention (one query row per sequence), split over the keys:
// CTA (row, head, split) covers a key chunk with 4 warps; in a warp, 8 keys at a time,
// 4 lanes per key each owning DH/4 head dimensions.  Partial (max, sum, output) per
// split go to a workspace and a second kernel merges them.
// ---------------------------------------------------------------------------
template <typename T, int DH>
__global__ void __launch_bounds__(128) attn_decode_split_kernel(const T* __restrict__ q, int ld_q, DevRange rows,
                                                                const int* row_tok, const int* tok_seq,
                                                                const int* tok_pos, const int* seq_len,
                                                                KVCacheView cache, int layer0, int n_heads, int causal,
                                                                float scale_log2, int chunk, int n_split,
                                                                float* ws) {
  PDL_ENTRY();
  constexpr int PD = DH / 4;   // dimensions per lane
  __shared__ float sm_m[4], sm_l[4];
  __shared__ float sm_o[4][DH];
  const int rh = blockIdx.x, split = blockIdx.y;
  const int r = rows.b() + rh / n_heads, h = rh % n_heads;
  if (r >= rows.e()) return;
  const int kvh = h / (n_heads / cache.n_kv_heads);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gk = lane >> 2, j = lane & 3;
  const int tok = row_tok[r];
  const int sq = tok_seq[tok], pos = tok_pos[tok];
  const int nk = causal ? pos + 1 : seq_len[sq];
  const int k_lo = split * chunk, k_hi = min(nk, k_lo + chunk);
  float* w = ws + ((size_t)rh * n_split + split) * (DH + 2);
  float qv[PD];
#pragma unroll
  for (int d = 0; d < PD; ++d) qv[d] = to_f(q[(size_t)r * ld_q + h * DH + j * PD + d]) * scale_log2;
  const T* Kp = (const T*)cache.k;
  const T* Vp = (const T*)cache.v;
  float m = -INFINITY, l = 0.f, o[PD];
#pragma unroll
  for (int d = 0; d < PD; ++d) o[d] = 0.f;
  for (int k0 = k_lo + warp * 8; k0 < k_hi; k0 += 32) {
    const int key = k0 + gk;
    const bool valid = key < k_hi;
    float sc = 0.f;
    size_t off = 0;
    if (valid) {
      off = cache.offset(layer0, sq, key, kvh) + j * PD;
#pragma unroll
      for (int d = 0; d < PD; ++d) sc = fmaf(qv[d], to_f(Kp[off + d]), sc);
    }
    sc += __shfl_xor_sync(0xffffffffu, sc, 1);
    sc += __shfl_xor_sync(0xffffffffu, sc, 2);
    if (!valid) sc = -INFINITY;
    float mx = sc;
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
    const float mn = fmaxf(m, mx);
    const float corr = (m == -INFINITY) ? 0.f : exp2f(m - mn);
    const float p = valid ? exp2f(sc - mn) : 0.f;
    float ps = p;
    ps += __shfl_xor_sync(0xffffffffu, ps, 4);
    ps += __shfl_xor_sync(0xffffffffu, ps, 8);
    ps += __shfl_xor_sync(0xffffffffu, ps, 16);
    l = l * corr + ps;
#pragma unroll
    for (int d = 0; d < PD; ++d) o[d] = o[d] * corr + (valid ? p * to_f(Vp[off + d]) : 0.f);
    m = mn;
  }
  // sum the 8 key groups of the warp
#pragma unroll
  for (int d = 0; d < PD; ++d) {
    o[d] += __shfl_xor_sync(0xffffffffu, o[d], 4);
    o[d] += __shfl_xor_sync(0xffffffffu, o[d], 8);
    o[d] += __shfl_xor_sync(0xffffffffu, o[d], 16);
  }
  if (lane == 0) {
    sm_m[warp] = m;
    sm_l[warp] = l;
  }
  if (gk == 0) {
#pragma unroll
    for (int d = 0; d < PD; ++d) sm_o[warp][j * PD + d] = o[d];
  }
  __syncthreads();
  float M = fmaxf(fmaxf(sm_m[0], sm_m[1]), fmaxf(sm_m[2], sm_m[3]));
  for (int d = tid; d < DH; d += 128) {
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (sm_m[k] != -INFINITY) acc += exp2f(sm_m[k] - M) * sm_o[k][d];
    w[d] = acc;
  }
  if (tid == 0) {
    float L = 0.f;
    for (int k = 0; k < 4; ++k)
      if (sm_m[k] != -INFINITY) L += exp2f(sm_m[k] - M) * sm_l[k];
    w[DH] = M;
    w[DH + 1] = L;
  }
}

template <typename T, int DH>
__global__ void attn_decode_combine_kernel(DevRange rows, int n_heads, int n_split, const float* ws, T* out,
                                           int ld_out) {
  PDL_ENTRY();
  const int rh = blockIdx.x;
  const int r = rows.b() + rh / n_heads, h = rh % n_heads;
  if (r >= rows.e()) return;
  const float* w = ws + (size_t)rh * n_split * (DH + 2);
  float M = -INFINITY;
  for (int s = 0; s < n_split; ++s) M = fmaxf(M, w[s * (DH + 2) + DH]);
  float L = 0.f;
  for (int s = 0; s < n_split; ++s) {
    const float ms = w[s * (DH + 2) + DH];
    if (ms != -INFINITY) L += exp2f(ms - M) * w[s * (DH + 2) + DH + 1];
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  for (int d = threadIdx.x; d < DH; d += blockDim.x) {
    float acc = 0.f;
    for (int s = 0; s < n_split; ++s) {
      const float ms = w[s * (DH + 2) + DH];
      if (ms != -INFINITY) acc += exp2f(ms - M) * w[s * (DH + 2) + d];
    }
    out[(size_t)r * ld_out + h * DH + d] = from_f<T>(acc * inv);
  }
}

template <typename T>
static void attn_dispatch(cudaStream_t st, const void* q, int ld_q, void* out, int ld_out, DevRange rows,
                          int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos,
                          const int* seq_len, KVCacheView cache, int layer0, int n_heads, int causal) {
  const int dh = cache.head_dim;
  const float scale = 1.f / sqrtf((float)dh);
  const int grid = cdiv(max_rows * n_heads, 8);
#define ATT_CASE(D)                                                                                         \
  case D:                                                                                                   \
    launch_k(attn_warp_kernel<T, D>, grid, 256, 0, st, (const T*)q, ld_q, (T*)out, ld_out, rows, row_tok, tok_seq, \
                                                 tok_pos, seq_len, cache, layer0, n_heads, causal, scale);  \
    break;
  switch (dh) {
    ATT_CASE(32)
    ATT_CASE(64)
    ATT_CASE(128)
    default:
      break;
  }
#undef ATT_CASE
}

// ---------------------------------------------------------------------------
// Generation-step attention (bf16): one query row per sequence, keys split into chunks of
// AD_CHUNK.  A CTA = (row, kv head, chunk): its K and V cache blocks (16 positions x
// head_dim, contiguous in the paged pool) are bulk-copied into shared memory on one
// mbarrier; per query head of the group the chunk's exact softmax partial (max m, sum l,
// sum p V) is formed in two passes over shared memory.  The last CTA of a (row, head) to
// finish (arrival counter) merges the chunk partials in chunk order and writes the output,
// then clears its counter for the next launch.
// ---------------------------------------------------------------------------
constexpr int AD_CHUNK = 128;
constexpr int AD_THREADS = 256;
constexpr int AD_WARPS = AD_THREADS / 32;
constexpr long long AD_TIMEOUT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz

__device__ __forceinline__ uint32_t ad_smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ bool ad_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(ad_smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool ad_try_wait_cluster(uint64_t* bar) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0;\nselp.u32 %0, 1, 0, "
      "p;\n}\n"
      : "=r"(ok)
      : "r"(ad_smem_u32(bar))
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool ad_wait(uint64_t* bar, unsigned* err) {
  if (ad_try_wait(bar, 0)) return true;
  const long long t0 = clock64();
  while (!ad_try_wait(bar, 0)) {
    if (clock64() - t0 > AD_TIMEOUT_CYCLES) {
      atomicOr(err, ERRW_TIMEOUT);
      return false;
    }
  }
  return true;
}

// CL: the chunks of a (token, kv head) form one thread-block cluster (n_split <= 8); every
// CTA pushes its chunk partials into the rank-0 CTA's shared memory (st.async, completing
// on its mbarrier), which merges them; otherwise partials go through global memory and the
// last CTA to arrive merges.
//
// CTAs are indexed by the step's token (not by its compacted row), so each CTA knows before
// the grid-dependency wait which cache blocks it reads: the blocks below the block of the
// token's own position were written by earlier steps (or the prompt pass) and are copied
// before the wait, overlapping the preceding kernels; the block holding the new key is
// copied after it.  The token's row among this layer's active rows is found after the wait;
// a token that left at an earlier layer lets its copies land and leaves.  The copy barrier
// takes two arrivals (before and after the wait), so it cannot complete between them.
//
// SV (one query head per KV head): the first half of the chunk's V rows has its own slots and
// the second half is copied into the K slots once the scores are formed, so a CTA holds 1.5
// chunks of rows instead of 2 (48 KB at d_h = 128): four CTAs fit on an SM and the grid of a
// 2-4 k-token context runs in one wave; the second half's copy overlaps the softmax and the
// first half's sum.
template <int DH, bool CL, bool SV>
__global__ void __launch_bounds__(AD_THREADS)
    attn_decode_kernel(const bf16* __restrict__ q, int ld_q, DevRange rows, const int* row_tok, const int* tok_seq,
                       const int* tok_pos, const int* seq_len, KVCacheView cache, int layer0, int n_heads, int causal,
                       float scale_log2, int n_split, float* __restrict__ ws, int* counters, bf16* __restrict__ out,
                       int ld_out, unsigned* err) {
  KT_BEGIN();
  constexpr int PARTS = DH / 8;                    // 16-byte pieces of a K / V row
  constexpr int KPI = 32 / PARTS;                  // keys per warp instruction
  constexpr int KIT = AD_CHUNK / (AD_WARPS * KPI); // key groups per warp
  extern __shared__ __align__(128) uint8_t ad_smem[];
  constexpr int HB = AD_CHUNK / 32;               // SV: cache blocks of the chunk's first half
  bf16* sK = reinterpret_cast<bf16*>(ad_smem);   // [AD_CHUNK][DH]; SV: then V rows HB*16..
  bf16* sV = sK + AD_CHUNK * DH;                  // [AD_CHUNK][DH]; SV: [AD_CHUNK / 2][DH]
  __shared__ __align__(8) uint64_t bar;
  __shared__ __align__(8) uint64_t bar2;          // SV: the second half of V
  __shared__ float s_p[AD_CHUNK];
  __shared__ float s_red[AD_THREADS / 32];
  __shared__ float s_o[AD_THREADS / 32][DH];
  __shared__ int s_last;
  __shared__ int s_row;
  __shared__ __align__(8) uint64_t red_bar;   // CL leader: the other chunks' partials
  constexpr int PW = DH + 4;                  // floats per pushed partial: o[DH], m, l, pad

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Hkv = cache.n_kv_heads, group = n_heads / Hkv;
  const int rk = blockIdx.x, split = blockIdx.y;
  const int t = rk / Hkv, kvh = rk - t * Hkv;   // the step's token t (its sequence and position
                                                // come from the pass's first kernel)
  const int sq = tok_seq[t], pos = tok_pos[t];
  const int nk = causal ? pos + 1 : seq_len[sq];
  const int n_eff = (nk + AD_CHUNK - 1) / AD_CHUNK;   // chunks holding keys of this token
  if (SV && group != 1) {   // (uniform over the grid) the K slots would be needed again
    if (tid == 0) atomicOr(err, ERRW_CONFIG);
    return;
  }
  if (!CL && split >= n_eff) return;   // (a cluster's CTAs all stay: they push empty partials)
  const int k_lo = split * AD_CHUNK, nkc = max(0, min(nk - k_lo, AD_CHUNK));
  const int nb = (nkc + 15) >> 4;                      // cache blocks of the chunk
  // blocks of the chunk below the block of the token's own position: written before this step
  const int n_pre = max(0, min(nb, (pos >> 4) - (k_lo >> 4)));
  float* sPart = reinterpret_cast<float*>(ad_smem + (SV ? 3 * AD_CHUNK / 2 : 2 * AD_CHUNK) * DH * 2);   // CL: [group][n_split][PW]
  constexpr int BLOCK_BYTES = 16 * DH * 2;
  KT_MARK(0);

  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 2;" ::"r"(ad_smem_u32(&bar)) : "memory");
    if (SV) asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(ad_smem_u32(&bar2)) : "memory");
    if (CL) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(ad_smem_u32(&red_bar)) : "memory");
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (CL && split == 0)
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(ad_smem_u32(&red_bar)),
                   "r"((uint32_t)(group * (n_split - 1) * PW * 4))
                   : "memory");
  }
  __syncthreads();
  // copy of block b of the chunk (b < nb) into its K slots and (V: !SV or b < HB) its V slots;
  // v_only (SV): block b >= HB's V rows into K slots (b - HB), completing on bar2
  auto copy_block = [&](int b, bool v_only) {
    const int bi = (k_lo >> 4) + b;
    int blk = (sq >= 0 && sq < cache.max_batch && bi < cache.max_blocks_per_seq)
                  ? cache.block_table[sq * cache.max_blocks_per_seq + bi]
                  : -1;
    if (blk < 0 || blk >= cache.n_blocks) {   // no reserved block: flag, copy block 0 (results unused)
      atomicOr(err, ERRW_POS);
      blk = 0;
    }
    const size_t off = (((size_t)layer0 * cache.n_blocks + blk) * Hkv + kvh) * (size_t)(16 * DH);
    if (SV && v_only) {
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                       ad_smem_u32(sK + (b - HB) * 16 * DH)),
                   "l"((const bf16*)cache.v + off), "r"((uint32_t)BLOCK_BYTES), "r"(ad_smem_u32(&bar2))
                   : "memory");
      return;
    }
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     ad_smem_u32(sK + b * 16 * DH)),
                 "l"((const bf16*)cache.k + off), "r"((uint32_t)BLOCK_BYTES), "r"(ad_smem_u32(&bar))
                 : "memory");
    if (!SV || b < HB)
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                       ad_smem_u32(sV + b * 16 * DH)),
                   "l"((const bf16*)cache.v + off), "r"((uint32_t)BLOCK_BYTES), "r"(ad_smem_u32(&bar))
                   : "memory");
  };
  // bytes of the phase-one copies of blocks [b0, b1)
  auto phase1_bytes = [&](int b0, int b1) {
    return (uint32_t)(((b1 - b0) + (SV ? max(0, min(b1, HB) - min(b0, HB)) : (b1 - b0))) * BLOCK_BYTES);
  };
  if (warp == 0) {
    if (lane == 0)
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(ad_smem_u32(&bar)),
                   "r"(phase1_bytes(0, n_pre))
                   : "memory");
    __syncwarp();
    if (lane < n_pre) copy_block(lane, false);
  }
  pdl_wait();
  KT_WAITED();
  pdl_launch_dependents();
  // this token's row among the layer's active rows (rows keep token order), or -1
  if (warp == 0) {
    const int rb = rows.b(), M = rows.e() - rb;
    int found = -1;
    for (int j0 = 0; j0 < M && found < 0; j0 += 32) {
      const int j = j0 + lane;
      const unsigned hit = __ballot_sync(0xffffffffu, j < M && row_tok[rb + j] == t);
      if (hit) found = rb + j0 + __ffs(hit) - 1;
    }
    if (lane == 0) s_row = found;
  }
  __syncthreads();
  const int r = s_row;
  if (warp == 0) {
    // second arrival: the block holding the new key (active tokens), or none
    if (lane == 0) {
      if (r >= 0)
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(ad_smem_u32(&bar)),
                     "r"(phase1_bytes(n_pre, nb))
                     : "memory");
      else
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(ad_smem_u32(&bar)) : "memory");
    }
    __syncwarp();
    if (r >= 0 && lane >= n_pre && lane < nb) copy_block(lane, false);
  }
  if (r < 0) {
    // the token left at an earlier layer (uniform over the cluster): let the copies land, leave
    if (warp == 0 && lane == 0) {
      bool ok = ad_wait(&bar, err);
      if (!ok) ad_wait(&bar, err);
    }
    __syncthreads();
    return;
  }
  const int slot = lane / PARTS, part = lane - slot * PARTS;
  // the first query head's piece (8 dims per lane), fetched while the cache blocks are in flight
  uint4 qraw = *reinterpret_cast<const uint4*>(q + (size_t)r * ld_q + kvh * group * DH + part * 8);
  // the leader's reduction barrier must be initialised before any CTA pushes to it: every
  // CTA arrives here (after the initialisation) and waits only just before its first push
  if (CL) asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  KT_MARK(1);
  {
    bool ok = ad_wait(&bar, err);
    if (!ok) ad_wait(&bar, err);   // second bounded wait for the copies in flight; results flagged
  }
  KT_MARK(2);

#pragma unroll 1
  for (int g = 0; g < group; ++g) {
    const int h = kvh * group + g;
    float qv[8];
    {
      const uint4 u = g == 0 ? qraw : *reinterpret_cast<const uint4*>(q + (size_t)r * ld_q + h * DH + part * 8);
      const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(b[i]);
        qv[2 * i] = f.x * scale_log2;
        qv[2 * i + 1] = f.y * scale_log2;
      }
    }
    // pass 1: scores of the warp's keys (all loads of the warp issued together)
    {
      uint4 kr[KIT];
#pragma unroll
      for (int it = 0; it < KIT; ++it)
        kr[it] = *reinterpret_cast<const uint4*>(sK + (warp * KPI + it * AD_WARPS * KPI + slot) * DH + part * 8);
      float d[KIT];
#pragma unroll
      for (int it = 0; it < KIT; ++it) {
        const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&kr[it]);
        float a = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 f = __bfloat1622float2(b[i]);
          a = fmaf(qv[2 * i], f.x, a);
          a = fmaf(qv[2 * i + 1], f.y, a);
        }
        d[it] = a;
      }
#pragma unroll
      for (int o = PARTS >> 1; o; o >>= 1)
#pragma unroll
        for (int it = 0; it < KIT; ++it) d[it] += __shfl_xor_sync(0xffffffffu, d[it], o);
      if (part == 0) {
#pragma unroll
        for (int it = 0; it < KIT; ++it) {
          const int key = warp * KPI + it * AD_WARPS * KPI + slot;
          s_p[key] = key < nkc ? d[it] : -INFINITY;
        }
      }
    }
    __syncthreads();
    KT_MARK(3);
    if (SV && nb > HB && warp == 0) {
      // every read of the K slots is done: the second half of V into them
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      if (lane == 0)
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(ad_smem_u32(&bar2)),
                     "r"((uint32_t)((nb - HB) * BLOCK_BYTES))
                     : "memory");
      __syncwarp();
      if (lane >= HB && lane < nb) copy_block(lane, true);
    }
    // chunk max, probabilities, chunk sum
    float mx = -INFINITY;
#pragma unroll
    for (int k = tid; k < AD_CHUNK; k += AD_THREADS) mx = fmaxf(mx, s_p[k]);
    mx = warp_max(mx);
    if (lane == 0) s_red[warp] = mx;
    __syncthreads();
    float M = s_red[0];
#pragma unroll
    for (int w = 1; w < AD_WARPS; ++w) M = fmaxf(M, s_red[w]);
    float ls = 0.f;
#pragma unroll
    for (int k = tid; k < AD_CHUNK; k += AD_THREADS) {
      const float pk = k < nkc ? exp2f(s_p[k] - M) : 0.f;
      s_p[k] = pk;
      ls += pk;
    }
    ls = warp_sum(ls);
    __syncthreads();   // every s_red[] read and s_p[] write done
    if (lane == 0) s_red[warp] = ls;
    KT_MARK(4);
    // pass 2: sum p V, lane = (key slot, 8 dims); keys past the chunk carry p = 0
    float o[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i] = 0.f;
    // key groups [it0, it1) of the warp (SV: the first half's groups read sV, the second's
    // the K slots after their copy has landed; key = ... + it * AD_WARPS * KPI, so groups below
    // KIT / 2 hold the keys below AD_CHUNK / 2)
    auto pv = [&](int it0, int it1, const bf16* base, int key0) {
      uint4 vr[KIT];
      float pr[KIT];
#pragma unroll
      for (int it = 0; it < KIT; ++it) {
        if (it < it0 || it >= it1) continue;
        const int key = warp * KPI + it * AD_WARPS * KPI + slot;
        vr[it] = *reinterpret_cast<const uint4*>(base + (key - key0) * DH + part * 8);
        pr[it] = s_p[key];
      }
#pragma unroll
      for (int it = 0; it < KIT; ++it) {
        if (it < it0 || it >= it1) continue;
        const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&vr[it]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 f = __bfloat1622float2(b[i]);
          // p == 0 for keys past the chunk (their V rows may hold anything, NaN included)
          o[2 * i] += pr[it] != 0.f ? pr[it] * f.x : 0.f;
          o[2 * i + 1] += pr[it] != 0.f ? pr[it] * f.y : 0.f;
        }
      }
    };
    if (!SV) {
      pv(0, KIT, sV, 0);
    } else {
      pv(0, KIT / 2, sV, 0);
      if (nb > HB) {
        bool ok = ad_wait(&bar2, err);
        if (!ok) ad_wait(&bar2, err);   // second bounded wait for the copies in flight; results flagged
        pv(KIT / 2, KIT, sK, AD_CHUNK / 2);
      }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int sft = PARTS; sft < 32; sft <<= 1) o[i] += __shfl_xor_sync(0xffffffffu, o[i], sft);
    if (slot == 0) {
#pragma unroll
      for (int i = 0; i < 8; ++i) s_o[warp][part * 8 + i] = o[i];
    }
    __syncthreads();
    const int rh = t * n_heads + h;
    if (CL) {
      if (g == 0) asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
      // chunk partial (empty chunk: m = -inf, l = 0, o = 0) -> slot [g][split] of the leader
      float* slot = sPart + ((size_t)g * n_split + split) * PW;
      for (int q4 = tid; q4 < PW / 4; q4 += AD_THREADS) {
        float4 v;
        float* vv = reinterpret_cast<float*>(&v);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int d = q4 * 4 + c;
          float sum = 0.f;
          if (d < DH) {
#pragma unroll
            for (int w = 0; w < AD_WARPS; ++w) sum += s_o[w][d];
          } else if (d == DH + 1) {
#pragma unroll
            for (int w = 0; w < AD_WARPS; ++w) sum += s_red[w];
          }
          vv[c] = nkc == 0 ? (d == DH ? -INFINITY : 0.f) : d == DH ? M : sum;
        }
        if (split == 0) {
          *reinterpret_cast<float4*>(slot + q4 * 4) = v;
        } else {
          uint32_t rd, rbar;
          asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(rd) : "r"(ad_smem_u32(slot + q4 * 4)));
          asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(rbar) : "r"(ad_smem_u32(&red_bar)));
          asm volatile(
              "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(rd),
              "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
              : "memory");
        }
      }
      __syncthreads();   // s_p / s_o / s_red reused by the next head of the group
      continue;
    }
    // chunk partial -> workspace [(row, head), split]: o[DH], m, l
    float* w = ws + ((size_t)rh * n_split + split) * (DH + 2);
    for (int d = tid; d < DH; d += AD_THREADS) {
      float sum = 0.f;
#pragma unroll
      for (int w2 = 0; w2 < AD_WARPS; ++w2) sum += s_o[w2][d];
      w[d] = sum;
    }
    if (tid == 0) {
      float sum = 0.f;
#pragma unroll
      for (int w2 = 0; w2 < AD_WARPS; ++w2) sum += s_red[w2];
      w[DH] = M;
      w[DH + 1] = sum;
    }
    __threadfence();
    __syncthreads();
    KT_MARK(5);
    if (tid == 0) s_last = atomicAdd(&counters[rh], 1) == n_eff - 1;
    __syncthreads();
    KT_MARK(6);
    if (s_last) {
      // last chunk of (row, head) to finish: merge the chunk partials in chunk order, every
      // load of the merge in flight at once
      __threadfence();
      const float* wb = ws + (size_t)rh * n_split * (DH + 2);
      const int d = tid;   // DH <= AD_THREADS
      // running merge over groups of 8 chunks (8 chunks' loads in flight at a time)
      float Mg = -INFINITY, L = 0.f, acc = 0.f;
      for (int c0 = 0; c0 < n_eff; c0 += 8) {
        float mc[8], lc[8], oc[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          mc[c] = -INFINITY;
          lc[c] = oc[c] = 0.f;
          if (c0 + c < n_eff) {
            const float* wc = wb + (size_t)(c0 + c) * (DH + 2);
            mc[c] = __ldcg(wc + DH);
            lc[c] = __ldcg(wc + DH + 1);
            oc[c] = d < DH ? __ldcg(wc + d) : 0.f;
          }
        }
        float Mn = Mg;
#pragma unroll
        for (int c = 0; c < 8; ++c) Mn = fmaxf(Mn, mc[c]);
        const float corr = Mg == -INFINITY ? 0.f : exp2f(Mg - Mn);
        L *= corr;
        acc *= corr;
#pragma unroll
        for (int c = 0; c < 8; ++c)
          if (c0 + c < n_eff) {
            const float sc = exp2f(mc[c] - Mn);
            L += sc * lc[c];
            acc += sc * oc[c];
          }
        Mg = Mn;
      }
      if (d < DH) out[(size_t)r * ld_out + h * DH + d] = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
      if (tid == 0) counters[rh] = 0;
    }
    __syncthreads();   // s_p / s_o / s_red reused by the next head of the group
  }
  if (CL && split == 0) {
    // leader: every chunk's partial is in shared memory -> merge in chunk order per head
    bool ok = false;
    {
      const long long t0 = clock64();
      while (!(ok = ad_try_wait_cluster(&red_bar))) {
        if (clock64() - t0 > 16 * AD_TIMEOUT_CYCLES) {
          atomicOr(err, ERRW_TIMEOUT);
          break;
        }
      }
    }
    if (!ok) return;
    for (int g = 0; g < group; ++g) {
      const int h = kvh * group + g;
      const float* sl = sPart + (size_t)g * n_split * PW;
      float Mg = -INFINITY;
      for (int c = 0; c < n_split; ++c) Mg = fmaxf(Mg, sl[c * PW + DH]);
      float L = 0.f, acc = 0.f;
      const int d = tid;
      for (int c = 0; c < n_split; ++c) {
        const float m = sl[c * PW + DH];
        if (m == -INFINITY) continue;
        const float sc = exp2f(m - Mg);
        L += sc * sl[c * PW + DH + 1];
        if (d < DH) acc += sc * sl[c * PW + d];
      }
      if (d < DH) out[(size_t)r * ld_out + h * DH + d] = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
    }
  }
}

static int g_attn_smem_set[2] = {0, 0};
static int g_ad_smem_set[8] = {0, 0, 0, 0, 0, 0, 0, 0};

void launch_attention(cudaStream_t st, int dt, const void* q, int ld_q, void* out, int ld_out, DevRange rows,
                      int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos, const int* seq_len,
                      KVCacheView cache, int layer0, int n_heads, int causal, int decode_keys, float* ws,
                      int* counters, unsigned* err, const int* key_exit, int kp_len, int q_rows, int n_layers) {
  if (max_rows <= 0) return;
  const int dh = cache.head_dim;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)dh);
  // prompt passes of bf16 models: the tcgen05 kernel when the caller gives the Q buffer's
  // extent and the pools' layer count (the mma.sync kernel below keeps the key mask of the
  // encoder's stop-entirely variant)
  if (decode_keys == 0 && dt == 1 && !key_exit && q_rows > 0 && n_layers > 0 &&
      launch_attention_tc(st, q, ld_q, q_rows, out, ld_out, rows, max_rows, row_tok, tok_seq, tok_pos, seq_len, cache,
                          n_layers, layer0, n_heads, causal, scale_log2, err) >= 0)
    return;
  if (decode_keys > 0 && ws && counters && dt == 1 && (dh == 64 || dh == 128) && cache.block_tokens == 16 &&
      (decode_keys + AD_CHUNK - 1) / AD_CHUNK <= ATTN_MAX_SPLIT && n_heads % cache.n_kv_heads == 0 &&
      n_heads / cache.n_kv_heads <= 8 &&
      ld_q % 8 == 0 && ((uintptr_t)q & 15) == 0) {
    const int n_split = (decode_keys + AD_CHUNK - 1) / AD_CHUNK;
    const dim3 grid(max_rows * cache.n_kv_heads, n_split);
    const int group = n_heads / cache.n_kv_heads;
    const bool cl = n_split > 1 && n_split <= 8;   // chunks of a (row, kv head) merged in a cluster
    const bool sv = group == 1;                     // one query head per KV head: 1.5 chunks of rows
    const int smem = (sv ? 3 * AD_CHUNK / 2 : 2 * AD_CHUNK) * dh * 2 + (cl ? group * n_split * (dh + 4) * 4 : 0);
    const int vi = (dh == 64 ? 0 : 4) + (cl ? 1 : 0) + (sv ? 2 : 0);
    void (*kern)(const bf16*, int, DevRange, const int*, const int*, const int*, const int*, KVCacheView, int, int, int,
                 float, int, float*, int*, bf16*, int, unsigned*) =
        vi == 0 ? attn_decode_kernel<64, false, false>
        : vi == 1 ? attn_decode_kernel<64, true, false>
        : vi == 2 ? attn_decode_kernel<64, false, true>
        : vi == 3 ? attn_decode_kernel<64, true, true>
        : vi == 4 ? attn_decode_kernel<128, false, false>
        : vi == 5 ? attn_decode_kernel<128, true, false>
        : vi == 6 ? attn_decode_kernel<128, false, true>
                  : attn_decode_kernel<128, true, true>;
    if (g_ad_smem_set[vi] < smem) {
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      g_ad_smem_set[vi] = smem;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(AD_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    int na = 0;
    if (cl) {
      at[na].id = cudaLaunchAttributeClusterDimension;
      at[na].val.clusterDim.x = 1;
      at[na].val.clusterDim.y = n_split;
      at[na].val.clusterDim.z = 1;
      ++na;
    }
    if (g_pdl) {
      at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      at[na].val.programmaticStreamSerializationAllowed = 1;
      ++na;
    }
    cfg.attrs = at;
    cfg.numAttrs = na;
    cudaLaunchKernelEx(&cfg, kern, (const bf16*)q, ld_q, rows, row_tok, tok_seq, tok_pos, seq_len, cache, layer0, n_heads,
                       causal, scale_log2, n_split, ws, counters, (bf16*)out, ld_out, err);
    return;
  }
  if (decode_keys > 0 && ws && (dh == 64 || dh == 128)) {
    // generation step: split the keys so that rows x heads x splits covers the GPU twice
    int n_split = (2 * 152 + max_rows * n_heads - 1) / (max_rows * n_heads);
    n_split = std::max(1, std::min(n_split, ATTN_MAX_SPLIT));
    int chunk = (decode_keys + n_split - 1) / n_split;
    chunk = std::max(32, ((chunk + 31) / 32) * 32);
    n_split = (decode_keys + chunk - 1) / chunk;
    dim3 grid(max_rows * n_heads, n_split);
#define DEC_CASE(T, D)                                                                                       \
  {                                                                                                          \
    launch_k(attn_decode_split_kernel<T, D>, grid, 128, 0, st, (const T*)q, ld_q, rows, row_tok, tok_seq, tok_pos, \
                                                         seq_len, cache, layer0, n_heads, causal, scale_log2, \
                                                         chunk, n_split, ws);                                \
    launch_k(attn_decode_combine_kernel<T, D>, max_rows * n_heads, 128, 0, st, rows, n_heads, n_split, ws, (T*)out, \
                                                                         ld_out);                           \
  }
    if (dt == 1) {
      if (dh == 64) DEC_CASE(bf16, 64) else DEC_CASE(bf16, 128)
    } else {
      if (dh == 64) DEC_CASE(float, 64) else DEC_CASE(float, 128)
    }
#undef DEC_CASE
    return;
  }
  if (dt == 1 && (dh == 64 || dh == 128)) {
    const int smem = 3 * 64 * (dh + 8) * 2;
    dim3 grid(cdiv(max_rows, 64), n_heads);
    if (dh == 64) {
      if (!g_attn_smem_set[0]) {
        cudaFuncSetAttribute(attn_prefill_mma_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        g_attn_smem_set[0] = 1;
      }
      launch_k(attn_prefill_mma_kernel<64>, grid, 128, smem, st, (const bf16*)q, ld_q, (bf16*)out, ld_out, rows, row_tok,
                                                           tok_seq, tok_pos, seq_len, cache, layer0, n_heads, causal,
                                                           scale_log2, key_exit, kp_len);
    } else {
      if (!g_attn_smem_set[1]) {
        cudaFuncSetAttribute(attn_prefill_mma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        g_attn_smem_set[1] = 1;
      }
      launch_k(attn_prefill_mma_kernel<128>, grid, 128, smem, st, (const bf16*)q, ld_q, (bf16*)out, ld_out, rows, row_tok,
                                                            tok_seq, tok_pos, seq_len, cache, layer0, n_heads, causal,
                                                            scale_log2, key_exit, kp_len);
    }
    return;
  }
  if (dt == 1)
    attn_dispatch<bf16>(st, q, ld_q, out, ld_out, rows, max_rows, row_tok, tok_seq, tok_pos, seq_len, cache, layer0,
                        n_heads, causal);
  else
    attn_dispatch<float>(st, q, ld_q, out, ld_out, rows, max_rows, row_tok, tok_seq, tok_pos, seq_len, cache, layer0,
                         n_heads, causal);
}

ADEPT_KTRACE_ATTACH(attention)

}  // namespace adept

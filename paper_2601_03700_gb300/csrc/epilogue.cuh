// GEMM epilogues applied to 32 consecutive output columns of one row.  Shared by the
// tcgen05 GEMM (a thread owns one accumulator row in tensor memory), the generation-step
// GEMM and the SIMT GEMM, so every path has one definition of each fused epilogue.
//
// Column layouts the epilogues rely on (fixed by the load-time repacking):
//  * RoPE families: inside each Q / K head the weight rows are interleaved so that
//    output columns (2i, 2i+1) hold the rotate-half pair (i, i + head_dim/2).
//  * SwiGLU: gate and up rows interleaved in blocks of 16, so a 32-column chunk
//    holds 16 gate and the matching 16 up columns.
#pragma once
#include "common.cuh"

namespace adept {

template <typename T> struct Vec16;
template <> struct Vec16<float> {
  static __device__ __forceinline__ void store(float* p, const float* v) {
    float4* q = reinterpret_cast<float4*>(p);
#pragma unroll
    for (int j = 0; j < 4; ++j) q[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  }
};
template <> struct Vec16<bf16> {
  static __device__ __forceinline__ void store(bf16* p, const float* v) {
    uint4 w[2];
    uint32_t* u = reinterpret_cast<uint32_t*>(w);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
      u[j] = *reinterpret_cast<uint32_t*>(&h);
    }
    uint4* q = reinterpret_cast<uint4*>(p);
    q[0] = w[0];
    q[1] = w[1];
  }
};

// 16 values to T* p (p 32-byte aligned for bf16, 64-byte for fp32).
template <typename T>
__device__ __forceinline__ void store16(T* p, const float* v) {
  Vec16<T>::store(p, v);
}

// Per-row facts the cache epilogues need: the token's position and the cache offset
// of its slot (-1 if the position has no reserved block); rope (optional): the row's
// (cos, sin) table row already staged by the caller.
struct EpiRow {
  long long cbase;
  int pos;
  const float2* rope;
};

__device__ __forceinline__ EpiRow epi_row(const Epi& e, int ra) {
  EpiRow r{-1, 0, nullptr};
  if (e.kind == EPI_QKV || e.kind == EPI_KV) {
    const int tok = e.row_tok[ra];
    r.pos = e.tok_pos[tok];
    r.cbase = e.cache.checked_base(e.layer0, e.tok_seq[tok], r.pos);
  }
  return r;
}

// Rotary embedding of 16 adjacent pairs (columns 2j, 2j+1 -> features i0+j, i0+j+half),
// written as two runs of 16 at dst[i0] and dst[i0 + half].
template <typename T>
__device__ __forceinline__ void rope_pairs(T* dst, int i0, int half, const float* v, const float2* tab) {
  float a[16], b[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float2 cs = tab[i0 + j];
    const float x1 = v[2 * j], x2 = v[2 * j + 1];
    a[j] = x1 * cs.x - x2 * cs.y;
    b[j] = x2 * cs.x + x1 * cs.y;
  }
  store16<T>(dst + i0, a);
  store16<T>(dst + i0 + half, b);
}

// A short tanh for the tanh form of GELU with bf16 results (its error stays far below the bf16
// rounding of the output): the hardware approximation tanh.approx.f32, relative error about
// 2^-11.
__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The activation of a 32-value chunk, switched once per chunk: a per-element switch in the
// unrolled loop would lay out 32 copies of every activation's code (for the epilogue warps of
// the tcgen05 GEMM, instruction fetch then dominated: GELU epilogues ran 5x slower than the
// others).  The tanh form of GELU with bf16 results uses tanh_approx; the rest keep tanhf / erff.
template <typename T>
__device__ __forceinline__ void act_chunk32(int act, float (&v)[32]) {
  constexpr bool fast = sizeof(T) == 2;
  if (act == ACT_GELU_TANH) {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float x = v[j], u = 0.79788456080286536f * (x + 0.044715f * x * x * x);
      v[j] = 0.5f * x * (1.f + (fast ? tanh_approx(u) : tanhf(u)));
    }
  } else if (act == ACT_GELU_ERF) {
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = gelu_erf_f(v[j]);
  } else if (act == ACT_TANH) {   // the encoder's pooler (one row per sequence): kept exact
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = tanhf(v[j]);
  }
}

// bias32 / resid32 (optional): the chunk's 32 bias values and the row's 32 residual
// values already staged by the caller (e.g. in shared memory) instead of e.bias[c0..] and
// e.resid[ra][c0..].  applied (EPI_APPLIED_* bits): what the caller has already done to v
// (bias and EPI_ACT activation; EPI_RESID residual).  KIND >= 0 fixes the epilogue kind at
// compile time (only its code is generated); -1 switches on e.kind.
template <typename T, int KIND = -1>
__device__ __forceinline__ void epi_chunk32(const Epi& e, int ra, int c0, int N, float (&v)[32], const EpiRow& rr,
                                            const float* bias32 = nullptr, const float* resid32 = nullptr,
                                            int applied = 0) {
  const bool full = c0 + 32 <= N;
  if (applied & EPI_APPLIED_BIAS_ACT) {
  } else if (bias32) {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (full || c0 + j < N) v[j] += bias32[j];
  } else if (e.bias) {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (full || c0 + j < N) v[j] += e.bias[c0 + j];
  }
  switch (KIND >= 0 ? KIND : e.kind) {
    case EPI_F32: {
      float* o = e.out_f32 + (size_t)ra * e.ld_f32 + c0;
      if (full && ((e.ld_f32 & 15) == 0)) {
        store16<float>(o, v);
        store16<float>(o + 16, v + 16);
      } else {
        for (int j = 0; j < 32; ++j)
          if (c0 + j < N) o[j] = v[j];
      }
      return;
    }
    case EPI_ACT: {
      if (!(applied & EPI_APPLIED_BIAS_ACT)) act_chunk32<T>(e.act, v);
      T* o = (T*)e.out_t + (size_t)ra * e.ld_t + c0;
      if (full && ((e.ld_t & 15) == 0)) {
        store16<T>(o, v);
        store16<T>(o + 16, v + 16);
      } else {
        for (int j = 0; j < 32; ++j)
          if (c0 + j < N) o[j] = from_f<T>(v[j]);
      }
      if (e.out_f32) {
        float* f = e.out_f32 + (size_t)ra * e.ld_f32 + c0;
        if (full && ((e.ld_f32 & 15) == 0)) {
          store16<float>(f, v);
          store16<float>(f + 16, v + 16);
        } else {
          for (int j = 0; j < 32; ++j)
            if (c0 + j < N) f[j] = v[j];
        }
      }
      return;
    }
    case EPI_RESID: {
      float* o = e.out_f32 + (size_t)ra * e.ld_f32 + c0;
      if (applied & EPI_APPLIED_RESID) {
        if (full && ((e.ld_f32 & 15) == 0)) {
          store16<float>(o, v);
          store16<float>(o + 16, v + 16);
        } else {
          for (int j = 0; j < 32; ++j)
            if (c0 + j < N) o[j] = v[j];
        }
        return;
      }
      const float* r = resid32 ? resid32 : e.resid + (size_t)ra * e.ld_resid + c0;
      if (full && ((e.ld_f32 & 15) == 0) && (resid32 || (e.ld_resid & 15) == 0)) {
        const float4* r4 = reinterpret_cast<const float4*>(r);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float4 x = r4[j];
          v[4 * j] += x.x;
          v[4 * j + 1] += x.y;
          v[4 * j + 2] += x.z;
          v[4 * j + 3] += x.w;
        }
        store16<float>(o, v);
        store16<float>(o + 16, v + 16);
      } else {
        for (int j = 0; j < 32; ++j)
          if (c0 + j < N) o[j] = r[j] + v[j];
      }
      return;
    }
    case EPI_SWIGLU: {
      float h[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) h[j] = silu_f(v[j]) * v[16 + j];
      T* o = (T*)e.out_t + (size_t)ra * e.ld_t + (c0 >> 1);
      if ((e.ld_t & 15) == 0) {
        store16<T>(o, h);
      } else {
        for (int j = 0; j < 16; ++j) o[j] = from_f<T>(h[j]);
      }
      return;
    }
    default:
      break;
  }
  // EPI_QKV / EPI_KV: [0, n_q) query, [n_q, n_q + n_kv) key, [n_q + n_kv, n_q + 2 n_kv) value.
  const int dh = e.head_dim, half = dh >> 1;
  const int nq = e.n_q_cols, nkv = e.n_kv_cols;
  if (c0 < nq) {
    const int h = c0 / dh, d0 = c0 % dh;
    T* q = (T*)e.out_t + (size_t)ra * e.ld_t + h * dh;
    if (e.rope) {
      rope_pairs<T>(q, d0 >> 1, half, v, rr.rope ? rr.rope : e.rope_table + (size_t)rr.pos * half);
    } else {
      store16<T>(q + d0, v);
      store16<T>(q + d0 + 16, v + 16);
    }
    return;
  }
  if (rr.cbase < 0) return;
  if (c0 < nq + nkv) {
    const int c = c0 - nq, h = c / dh, d0 = c % dh;
    T* k = (T*)e.cache.k + rr.cbase + (size_t)h * e.cache.head_stride();
    if (e.rope) {
      rope_pairs<T>(k, d0 >> 1, half, v, rr.rope ? rr.rope : e.rope_table + (size_t)rr.pos * half);
    } else {
      store16<T>(k + d0, v);
      store16<T>(k + d0 + 16, v + 16);
    }
    return;
  }
  {
    const int c = c0 - nq - nkv, h = c / dh, d0 = c % dh;
    T* vv = (T*)e.cache.v + rr.cbase + (size_t)h * e.cache.head_stride() + d0;
    store16<T>(vv, v);
    store16<T>(vv + 16, v + 16);
  }
}

}  // namespace adept

// Stream-K weight-streaming GEMM for sm_103a: C[M, N] = A[M, K] * W[N, K]^T with M <= 16.
//
// A generation step at batch 1 multiplies every weight once (2 flops per weight byte), so the
// step's GEMMs are a stream over W and their time is W's bytes over the HBM bandwidth, plus
// whatever part of the stream the kernel leaves idle.  This kernel keeps every SM streaming
// until the end:
//
//  * Work: the output features are cut into 32-feature tiles and K into 256-wide blocks; a
//    (tile, k-block) unit is 16 KB of weights.  One CTA per SM takes an equal contiguous
//    share of the units in tile-major order (stream-K), so no SM idles at the end of a
//    launch while others finish a last tile.
//  * Ring: one producer warp issues a cp.async.bulk.tensor copy per unit into a ring of
//    16 KB slots, completing on the slot's full barrier; four consumer warps release a slot
//    through its empty barrier (one arrival per warp), so a warp never waits for the other
//    warps before the producer can refill.  Weights do not depend on the preceding kernel,
//    so the first slots are issued before the programmatic-dependent-launch wait.
//  * One CTA per SM: the CTA takes just over half an SM's shared memory.  Consecutive
//    launches overlap (their CTAs are placed wherever there is room), and two CTAs of this
//    kernel on one SM would each stream at half rate while another SM idles, so the launch's
//    equal shares would end at twice the time; a five-slot ring leaves room beside the CTA
//    for one CTA of the neighbouring kernels (attention, cluster K-split GEMM).
//  * A operand: after the wait the launch's token rows (all of K) are staged once in shared
//    memory, copied (bf16) or standardised from the fp32 residual stream with row statistics
//    computed here or handed over by the producer of the rows.  A QKV launch of a generation step
//    may first take the previous layer's exit step (ds_exit_stage): its kept rows, standardised,
//    are then the operand.
//  * MMA: mma.sync m16n8k16 with the weight features as the m16 operand and the token rows
//    as the n8 operand (the contraction is far below the tensor-core ridge; only bytes count).
//  * Split tiles: a tile shared by several CTAs is finished by the last one to arrive: each
//    contributor writes its fp32 partial tile to its own slot, then increments the tile's
//    counter; the CTA that sees the final count sums the partials in contributor order (the
//    same sum every run), applies the fused epilogue and resets the counter.  No CTA waits for
//    another.
//  * Every mbarrier wait is bounded (ring waits by the runtime wait limit, the drain of copies
//    in flight by a fixed, longer one); on time-out the CTA records ERRW_TIMEOUT, stops, and
//    waits for its copies in flight before it exits.
#define ADEPT_TU_ID 8
#include "gemm_stream.h"
#include "epilogue.cuh"
#include "gemm_tc.h"
#include "kernels.h"

#include <cuda.h>

#include <algorithm>
#include <cstring>

namespace adept {
namespace {

constexpr int DS_BN = 32;                         // output features per tile
constexpr int DS_KB = 256;                        // k per unit
constexpr int DS_CHUNK = DS_BN * 128;             // one [32 rows][64 k] 128-byte-swizzled chunk
constexpr int DS_STAGE = DS_BN * DS_KB * 2;       // 16 KB per unit
constexpr int DS_NC = 4;                          // MMA (consumer) warps
constexpr int DS_NE = 2;                          // epilogue warps
constexpr int DS_WARPS = 1 + DS_NC + DS_NE;       // + the producer warp
constexpr int DS_THREADS = 32 * DS_WARPS;
constexpr int DS_MAX_STAGES = 12;
constexpr int DS_RING_STAGES = 5;                 // ring depth (measured at the Llama-7B shapes: 3-7 tried)
constexpr int DS_RP = DS_BN + 1;                  // floats per token row of a partial tile
constexpr int DS_MAXG = 32;                       // problems of a grouped launch (one warp's lanes)
static_assert(DS_MAXG <= 32, "the row counts of a launch are read by one warp");
constexpr int DS_SMEM_LIMIT = 200 * 1024;
constexpr long long DS_TIMEOUT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz
constexpr long long DS_MIN_STREAM_BYTES = 8ll << 20;    // below: the cluster K-split kernel
constexpr int DS_MIN_N = 8192;                           // single problems narrower: the cluster kernel
enum : int { DS_STATS_HERE = 0, DS_STATS_ROWS = 1, DS_STATS_TILES = 2 };

template <int MAXG>
struct DsParams {
  CUtensorMap wmap[MAXG];   // W as {64, N, K/64}, box {64, 32, 4}, 128-byte swizzle
  const uint8_t* bt[MAXG];  // tile-contiguous copy of W (GemmProblem::Bt) or NULL: the unit of
                            // (tile t, k-block kb) is the 16 KB at bt + (t * nkb + kb) * 16 KB
  DevRange rows[MAXG];
  Epi epi[MAXG];
  int n_probs;
  int grouped;        // 1: the units are partitioned over the problems with rows, after the wait
  int tiles, nkb, N, K;
  int stages;
  int max_m;
  int arows;          // A rows held in shared memory
  int apitch;         // A row pitch in elements
  int off_a, off_p;   // dynamic shared-memory offsets (from the 1024-aligned base)
  const bf16* A;
  int lda;
  const float* X;     // fused standardisation source
  int ldx;
  const int* in_rows;
  int norm_mode;
  float eps;
  int fused_norm;
  int stat_mode;
  const float2* row_stats;
  const float2* tile_stats;
  int n_stiles;
  float* part;
  int* cnt;
  unsigned* err;
  SpanCtx span;
  int exit_on;   // EPI_QKV, one problem: the previous layer's exit step first (ex)
  DsExit ex;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait: `limit` is the runtime wait limit for pipeline progress, DS_TIMEOUT_CYCLES for
// the drain of copies in flight.
__device__ __forceinline__ bool ds_wait(uint64_t* bar, uint32_t parity, unsigned* err, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > limit) {
      atomicOr(err, ERRW_TIMEOUT);
      return false;
    }
  }
  return true;
}
__device__ __forceinline__ void tma_load_3d(const CUtensorMap* tm, uint64_t* bar, void* dst, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::
          "r"(smem_u32(dst)),
      "l"((uint64_t)tm), "r"(0), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}
// 1-D bulk copy of `bytes` contiguous bytes (16-byte aligned, a multiple of 16), completing on bar.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t ld_shared_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Barrier of the epilogue warps only (producer and MMA warps keep streaming meanwhile).
__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, %0;" ::"n"(DS_NE * 32) : "memory"); }

// Stream-K partition of U units over G CTAs: CTA c takes [start(c), start(c + 1)).
__device__ __forceinline__ long long ds_start(long long c, long long U, long long G) { return c * U / G; }
// The CTA whose range holds unit u (the last CTA c with start(c) <= u).
__device__ __forceinline__ long long ds_owner(long long u, long long U, long long G) {
  return ((u + 1) * G + U - 1) / U - 1;
}

// Fused epilogue of one tile, element-parallel over the epilogue warps: warp ew takes rows
// ew, ew + DS_NE, ..., lane = feature.
template <int KIND>
__device__ __forceinline__ void ds_epilogue(const Epi& e, const float* sS, int M, int rb, int f0, int N, int ew,
                                            int lane, const int* s_pos, const int* s_blk) {
  for (int row = ew; row < M; row += DS_NE) {
    const int ra = rb + row, c = f0 + lane;
    const bool valid = c < N;
    float v = sS[row * DS_RP + lane];
    if (e.bias && valid) v += e.bias[c];
    if (KIND == EPI_F32) {
      if (valid) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
    } else if (KIND == EPI_ACT) {
      v = apply_act(e.act, v);
      if (valid) {
        ((bf16*)e.out_t)[(size_t)ra * e.ld_t + c] = __float2bfloat16_rn(v);
        if (e.out_f32) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
      }
    } else if (KIND == EPI_RESID) {
      if (valid) v += e.resid[(size_t)ra * e.ld_resid + c];
      if (valid) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
      if (e.tile_stats) {   // (mean, M2) of the row's 32 results (full tiles: N % 32 == 0)
        const float mean = warp_sum(v) * (1.f / DS_BN);
        const float m2 = warp_sum((v - mean) * (v - mean));
        if (lane == 0) e.tile_stats[(size_t)ra * (N / DS_BN) + f0 / DS_BN] = make_float2(mean, m2);
      }
    } else if (KIND == EPI_SWIGLU) {
      // features interleaved in blocks of 16: lanes 0-15 gate, 16-31 the matching up
      const float u = __shfl_down_sync(0xffffffffu, v, 16);
      if (lane < 16) ((bf16*)e.out_t)[(size_t)ra * e.ld_t + (f0 >> 1) + lane] = __float2bfloat16_rn(silu_f(v) * u);
    } else {   // EPI_QKV / EPI_KV: q -> out_t, k / v -> the row's cache slot; RoPE pairs adjacent
      const KVCacheView& cv = e.cache;
      const int pos = s_pos[row], blk = s_blk[row];
      EpiRow rr;
      rr.pos = blk < 0 ? 0 : pos;   // an invalid position (flagged by the pass) reads a valid table row
      rr.cbase = blk < 0 ? -1
                         : (long long)((((size_t)e.layer0 * cv.n_blocks + blk) * cv.n_kv_heads) * cv.block_tokens +
                                       (pos % cv.block_tokens)) *
                               cv.head_dim;
      const int dh = e.head_dim, half = dh >> 1, nq = e.n_q_cols, nkv = e.n_kv_cols;
      const int base = c < nq ? 0 : c < nq + nkv ? nq : nq + nkv;
      const int hd = (c - base) / dh, d = (c - base) - hd * dh;
      const float pv = __shfl_xor_sync(0xffffffffu, v, 1);   // the other member of the pair
      float o = v;
      int od = d;
      if (e.rope && base < nq + nkv) {
        const int ip = d >> 1;
        const float2 cs = e.rope_table[(size_t)rr.pos * half + ip];
        o = (d & 1) ? v * cs.x + pv * cs.y : v * cs.x - pv * cs.y;
        od = (d & 1) ? ip + half : ip;
      }
      if (valid) {
        if (base == 0 && nq > 0) {
          ((bf16*)e.out_t)[(size_t)ra * e.ld_t + hd * dh + od] = __float2bfloat16_rn(o);
        } else if (rr.cbase >= 0) {
          bf16* dst = (bf16*)(base == nq ? e.cache.k : e.cache.v);
          dst[rr.cbase + (size_t)hd * e.cache.head_stride() + od] = __float2bfloat16_rn(o);
        }
      }
    }
  }
}

// Stages rows 0..Ms-1 of the A operand into sA (bf16, pitch apitch; all K), rows
// Ms..arows-1 zero.  All threads of the CTA take part; one round trip to memory: a plain bf16
// operand is copied with cp.async; a standardised one is read into registers (two rows at a
// time, DS_XV float4 per thread and row) while its row statistics are loaded (or reduced from
// those registers), then written standardised.
constexpr int DS_XV = 5;    // float4 per thread and row: rows up to DS_XV * 4 * DS_THREADS floats
template <int MAXG>
__device__ void ds_stage_a(const DsParams<MAXG>& p, bf16* sA, int Ms, float* s_mu, float* s_rs,
                           float (*s_red)[16]) {   // s_red: [DS_WARPS][16]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, K = p.K, ap = p.apitch;
  for (int i = tid; i < (p.arows - Ms) * (ap >> 3); i += DS_THREADS) {   // zero rows past Ms
    const int r = Ms + i / (ap >> 3), c = i % (ap >> 3);
    *reinterpret_cast<uint4*>(sA + (size_t)r * ap + c * 8) = make_uint4(0, 0, 0, 0);
  }
  if (!p.fused_norm) {
    const int cpr = K >> 3;
    for (int i = tid; i < Ms * cpr; i += DS_THREADS) {
      const int r = i / cpr, c = i - r * cpr;
      cp_async16(sA + (size_t)r * ap + c * 8, p.A + (size_t)r * p.lda + c * 8);
    }
    cp_async_wait_all();
    __syncthreads();
    return;
  }
  const int K4 = K >> 2;
  for (int r0 = 0; r0 < Ms; r0 += 2) {
    const int nr = min(2, Ms - r0);
    float4 xv[2][DS_XV];
    const float* xr[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int r = k < nr ? r0 + k : r0;
      xr[k] = p.X + (size_t)(p.in_rows ? p.in_rows[r] : r) * p.ldx;
    }
    // the rows' values: every load issued before any is used
#pragma unroll
    for (int k = 0; k < 2; ++k)
#pragma unroll
      for (int j = 0; j < DS_XV; ++j) {
        const int v = tid + j * DS_THREADS;
        xv[k][j] = (k < nr && v < K4) ? *reinterpret_cast<const float4*>(xr[k] + v * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    if (p.stat_mode == DS_STATS_ROWS) {
      if (tid < nr) {
        const float2 st = p.row_stats[r0 + tid];
        s_mu[r0 + tid] = st.x;
        s_rs[r0 + tid] = st.y;
      }
    } else if (p.stat_mode == DS_STATS_TILES) {
      // the row's moments from the producer's 32-column (mean, M2) tiles, about the first
      // tile's mean c: S1 = sum 32 (m_t - c), S2 = sum M2_t + 32 (m_t - c)^2 (warp k: row r0 + k)
      if (warp < nr) {
        const int r = r0 + warp;
        const float2* ts = p.tile_stats + (size_t)r * p.n_stiles;
        const float c = ts[0].x;
        float s1 = 0.f, s2 = 0.f;
        for (int t = lane; t < p.n_stiles; t += 32) {
          const float2 b = ts[t];
          const float dm = b.x - c;
          s1 += 32.f * dm;
          s2 += b.y + 32.f * dm * dm;
        }
        s1 = warp_sum(s1);
        s2 = warp_sum(s2);
        if (lane == 0) {
          const float dmean = s1 / K, var = fmaxf(s2 / K - dmean * dmean, 0.f), mean = c + dmean;
          float mu = 0.f, rs = 1.f;
          if (p.norm_mode == NORM_LN) {
            mu = mean;
            rs = rsqrtf(var + p.eps);
          } else if (p.norm_mode == NORM_RMS) {
            rs = rsqrtf(var + mean * mean + p.eps);
          }
          s_mu[r] = mu;
          s_rs[r] = rs;
        }
      }
    } else {
      // statistics of the rows in registers: mean (LayerNorm), then the centred second moment
      float mu[2] = {0.f, 0.f};
      if (p.norm_mode == NORM_LN) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          float a = 0.f;
#pragma unroll
          for (int j = 0; j < DS_XV; ++j) a += (xv[k][j].x + xv[k][j].y) + (xv[k][j].z + xv[k][j].w);
          a = warp_sum(a);
          if (lane == 0) s_red[warp][k] = a;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          float t = 0.f;
          for (int w = 0; w < DS_WARPS; ++w) t += s_red[w][k];
          mu[k] = t / K;
        }
        __syncthreads();
      }
      if (p.norm_mode != NORM_COPY) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          float a = 0.f;
#pragma unroll
          for (int j = 0; j < DS_XV; ++j) {
            const int v = tid + j * DS_THREADS;
            if (v < K4) {
              const float4 x = xv[k][j];
              const float c0 = x.x - mu[k], c1 = x.y - mu[k], c2 = x.z - mu[k], c3 = x.w - mu[k];
              a += (c0 * c0 + c1 * c1) + (c2 * c2 + c3 * c3);
            }
          }
          a = warp_sum(a);
          if (lane == 0) s_red[warp][k] = a;
        }
        __syncthreads();
        if (tid < nr) {
          float t = 0.f;
          for (int w = 0; w < DS_WARPS; ++w) t += s_red[w][tid];
          s_mu[r0 + tid] = mu[tid];
          s_rs[r0 + tid] = rsqrtf(t / K + p.eps);
        }
      } else if (tid < nr) {
        s_mu[r0 + tid] = 0.f;
        s_rs[r0 + tid] = 1.f;
      }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      if (k >= nr) break;
      const int r = r0 + k;
      const float mu = s_mu[r], rs = s_rs[r];
#pragma unroll
      for (int j = 0; j < DS_XV; ++j) {
        const int v = tid + j * DS_THREADS;
        if (v < K4) {
          const float4 x = xv[k][j];
          const __nv_bfloat162 lo = __floats2bfloat162_rn((x.x - mu) * rs, (x.y - mu) * rs);
          const __nv_bfloat162 hi = __floats2bfloat162_rn((x.z - mu) * rs, (x.w - mu) * rs);
          uint2 u;
          u.x = *reinterpret_cast<const uint32_t*>(&lo);
          u.y = *reinterpret_cast<const uint32_t*>(&hi);
          *reinterpret_cast<uint2*>(sA + (size_t)r * ap + v * 4) = u;
        }
      }
    }
    __syncthreads();
  }
}

// What the exit step reads before the grid-dependency wait: everything the previous layer's exit
// step wrote (it finished several launches earlier), i.e. the layer's row count and exit count,
// the threshold, the first row's token, forced layer and inertia (from HBM by now); only s_i
// (the preceding kernel's output) is read after the wait.
struct DsExitPre {
  float4 xi[DS_XV];
  int n, base, tok0, f0;
  float delta;
};
template <int MAXG>
__device__ __forceinline__ void ds_exit_prefetch(const DsParams<MAXG>& p, DsExitPre& e) {
  const DsExit& x = p.ex;
  const int tid = threadIdx.x, K4 = p.K >> 2;
  e.n = x.ctr[CTR_ACTIVE + x.par];
  e.base = x.ctr[CTR_PREFIX + x.layer - 1];
  e.delta = *x.delta;
  e.tok0 = x.row_tok[0];
  e.f0 = (x.forced && tid == 0) ? x.forced[e.tok0] : 0;
  const float4* i4 = reinterpret_cast<const float4*>(x.I);
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int j = 0; j < DS_XV; ++j) {
    const int v = tid + j * DS_THREADS;
    e.xi[j] = (v < K4 && !x.first) ? i4[v] : z4;
  }
}

// The previous layer's exit step inside the QKV launch (DsExit; the global similarity of Sec.
// 4.1), rows one at a time: s_i and the inertia read once into registers, the four sums reduced
// over the CTA in a fixed order (every CTA of the launch decides alike), the decision (a forced
// layer, else similarity >= delta), then from the registers the kept row standardised into the A
// operand at its compacted index, and this CTA's slice of the moved rows (a leaving row's s_{i-1}
// copied from memory).  Rows past the kept ones are zeroed.  Ends with a CTA barrier; s_M /
// s_live / s_nlive describe the kept rows.
template <int MAXG>
__device__ void ds_exit_stage(const DsParams<MAXG>& p, const DsExitPre& pre, bf16* sA, float (*s_red)[16], int* s_M,
                              int* s_live, int* s_nlive, int* s_tokk, float* s_bc) {
  const DsExit& x = p.ex;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int K = p.K, K4 = K >> 2, ap = p.apitch;
  const int G = gridDim.x, c = blockIdx.x;
  const int n_all = pre.n;
  const int n = min(n_all, p.max_m);
  const int base = pre.base;
  const float delta = pre.delta;
  if (n_all > p.max_m && c == 0 && tid == 0) atomicOr(x.err, ERRW_CONFIG);
  // this CTA's slice of every moved row: float4 indices [v0, v1)
  const int v0 = (int)((long long)c * K4 / G), v1 = (int)((long long)(c + 1) * K4 / G);
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
  int k = 0, e = 0;   // rows kept / left so far (the same in every thread)
  for (int r = 0; r < n; ++r) {
    const float4* s4 = reinterpret_cast<const float4*>(x.Xout + (size_t)r * K);
    const float4* i4 = reinterpret_cast<const float4*>(x.I + (size_t)r * K);
    const float4* p4 = reinterpret_cast<const float4*>(x.Xin + (size_t)r * K);
    const int tok = r == 0 ? pre.tok0 : x.row_tok[r];
    float4 xs[DS_XV], xi[DS_XV];
#pragma unroll
    for (int j = 0; j < DS_XV; ++j) {   // every load first (the first row's inertia: read before the wait)
      const int v = tid + j * DS_THREADS;
      xs[j] = v < K4 ? s4[v] : z4;
      xi[j] = r == 0 ? pre.xi[j] : (v < K4 && !x.first) ? i4[v] : z4;
    }
    float ns = 0.f, ni = 0.f, dot = 0.f, sx = 0.f;
#pragma unroll
    for (int j = 0; j < DS_XV; ++j) {
      const float4 a = xs[j], b = xi[j];
      ns += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
      ni += b.x * b.x + b.y * b.y + b.z * b.z + b.w * b.w;
      dot += a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w;
      sx += a.x + a.y + a.z + a.w;
    }
    ns = warp_sum(ns);
    ni = warp_sum(ni);
    dot = warp_sum(dot);
    sx = warp_sum(sx);
    if (lane == 0) {
      s_red[warp][0] = ns;
      s_red[warp][1] = ni;
      s_red[warp][2] = dot;
      s_red[warp][3] = sx;
    }
    __syncthreads();
    if (tid == 0) {
      float a = 0.f, b = 0.f, cc = 0.f, m = 0.f;
      for (int w = 0; w < DS_WARPS; ++w) {
        a += s_red[w][0];
        b += s_red[w][1];
        cc += s_red[w][2];
        m += s_red[w][3];
      }
      int ex = 0;
      if (x.test) {
        const float cs = exit_similarity(EXIT_GLOBAL, a, b, cc, 0.f, 0.f);
        if (x.sim && c == 0) x.sim[(size_t)tok * x.n_layers + (x.layer - 1)] = cs;
        const int f = r == 0 ? pre.f0 : x.forced ? x.forced[tok] : 0;
        if (f != 0 && (f < 2 || f > x.n_layers) && c == 0) atomicOr(x.err, ERRW_FORCED);
        ex = (f > 0) ? (f == x.layer) : (cs >= delta);
      }
      s_bc[0] = ex ? 1.f : 0.f;
      s_bc[1] = a > 0.f ? rsqrtf(a) : 0.f;                 // inertia step weight 1 / |s_i|
      s_bc[2] = x.norm_mode == NORM_LN ? m / K : 0.f;       // the row's mean (LayerNorm)
      s_bc[3] = a;                                          // sum of squares (RMSNorm)
    }
    __syncthreads();
    const bool left = s_bc[0] != 0.f;
    const float w = s_bc[1], mu = s_bc[2];
    if (!left) {
      // the kept row standardised (as the standardisation kernel: LayerNorm two-pass from the
      // registers, RMSNorm from the sum of squares) into A row k, bf16
      float rs = 1.f, m0 = 0.f;
      if (x.norm_mode == NORM_LN) {
        float c2 = 0.f;
#pragma unroll
        for (int j = 0; j < DS_XV; ++j)
          if (tid + j * DS_THREADS < K4) {
            const float4 a = xs[j];
            c2 += (a.x - mu) * (a.x - mu) + (a.y - mu) * (a.y - mu) + (a.z - mu) * (a.z - mu) +
                  (a.w - mu) * (a.w - mu);
          }
        c2 = warp_sum(c2);
        if (lane == 0) s_red[warp][6] = c2;
        __syncthreads();
        float t = 0.f;
        for (int w2 = 0; w2 < DS_WARPS; ++w2) t += s_red[w2][6];
        rs = rsqrtf(t / K + x.eps);
        m0 = mu;
      } else if (x.norm_mode == NORM_RMS) {
        rs = rsqrtf(s_bc[3] / K + x.eps);
      }
      float4* xn = reinterpret_cast<float4*>(x.Xnext + (size_t)k * K);
      float4* in = reinterpret_cast<float4*>(x.Inext + (size_t)k * K);
#pragma unroll
      for (int j = 0; j < DS_XV; ++j) {
        const int v = tid + j * DS_THREADS;
        if (v < K4) {
          const float4 a = xs[j], b = xi[j];
          const __nv_bfloat162 lo = __floats2bfloat162_rn((a.x - m0) * rs, (a.y - m0) * rs);
          const __nv_bfloat162 hi = __floats2bfloat162_rn((a.z - m0) * rs, (a.w - m0) * rs);
          uint2 u;
          u.x = *reinterpret_cast<const uint32_t*>(&lo);
          u.y = *reinterpret_cast<const uint32_t*>(&hi);
          *reinterpret_cast<uint2*>(sA + (size_t)k * ap + v * 4) = u;
          if (v >= v0 && v < v1) {
            xn[v] = a;
            in[v] = make_float4(b.x + a.x * w, b.y + a.y * w, b.z + a.z * w, b.w + a.w * w);
          }
        }
      }
      if (tid == 0) {
        s_tokk[k] = tok;
        if (c == 0) x.row_tok_next[k] = tok;
      }
      ++k;
    } else {
      // the leaving row's mapper inputs at its exit slot
      const size_t slot = (size_t)(base + e);
      float4* hs = reinterpret_cast<float4*>(x.hsm_s + slot * K);
      float4* hp = reinterpret_cast<float4*>(x.hsm_prev + slot * K);
      float4* hi = reinterpret_cast<float4*>(x.hsm_I + slot * K);
#pragma unroll
      for (int j = 0; j < DS_XV; ++j) {
        const int v = tid + j * DS_THREADS;
        if (v < K4 && v >= v0 && v < v1) {
          hs[v] = xs[j];
          hp[v] = p4[v];
          hi[v] = xi[j];
        }
      }
      if (tid == 0 && c == 0) {
        x.exit_tok[base + e] = tok;
        if (x.exit_layer) x.exit_layer[tok] = x.layer;
      }
      ++e;
    }
    __syncthreads();   // s_red / s_bc are reused by the next row
  }
  // rows past the kept ones stay zero (they feed only token columns that are never stored)
  for (int i = tid; i < (p.arows - k) * (ap >> 3); i += DS_THREADS) {
    const int rr = k + i / (ap >> 3), cc = i % (ap >> 3);
    *reinterpret_cast<uint4*>(sA + (size_t)rr * ap + cc * 8) = make_uint4(0, 0, 0, 0);
  }
  if (tid == 0) {
    if (c == 0) {
      x.ctr[CTR_ACTIVE + (x.par ^ 1)] = k;
      x.ctr[CTR_EXITED] = base + e;
      x.ctr[CTR_PREFIX + x.layer] = base + e;
    }
    s_M[0] = k;
    s_live[0] = 0;
    *s_nlive = k > 0 ? 1 : 0;
  }
  __syncthreads();
}

// MB: 8-token blocks of the A operand (1: M <= 8, 2: M <= 16); KIND: the epilogue kind.
template <int MB, int KIND, int MAXG>
__global__ void __launch_bounds__(DS_THREADS, 2) gemm_stream_kernel(const __grid_constant__ DsParams<MAXG> p) {
  KT_BEGIN();
  extern __shared__ __align__(128) uint8_t ds_smem_raw[];
  __shared__ __align__(8) uint64_t full[DS_MAX_STAGES];
  __shared__ __align__(8) uint64_t empty[DS_MAX_STAGES];
  __shared__ __align__(8) uint64_t tb_full[2], tb_empty[2];   // tile hand-off, MMA warps -> epilogue warps
  __shared__ float s_mu[16], s_rs[16];
  __shared__ float s_red[DS_WARPS][16];
  __shared__ int s_live[MAXG];     // problems with rows, in order
  __shared__ int s_M[MAXG], s_rb[MAXG];
  __shared__ int s_nlive, s_last;
  __shared__ int s_pos[16], s_blk[16];   // cache epilogues: each row's position and cache block
  __shared__ int s_tokk[16];             // exit step: the kept rows' tokens
  __shared__ float s_bc[4];              // exit step: one row's decision, weight, mean, sum of squares
  __shared__ int s_info[2][3];           // per hand-off buffer: live problem slot, tile, whole
  __shared__ int s_eok[DS_NE];           // epilogue warps: still following the hand-offs
  __shared__ unsigned s_span_left;
  __shared__ unsigned long long s_span_t0;
  SpanScope span(p.span, &s_span_left, &s_span_t0);

  const long long wlim = wait_limit();   // the runtime wait limit, read once
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint8_t* smem = ds_smem_raw + ((1024 - (smem_u32(ds_smem_raw) & 1023)) & 1023);
  uint8_t* sW = smem;                                           // [S][4 chunks][32 rows][128 B], swizzled
  bf16* sA = reinterpret_cast<bf16*>(smem + p.off_a);           // [arows][apitch]
  float* sT = reinterpret_cast<float*>(smem + p.off_p);         // [2][16][DS_RP] tile hand-off buffers
  const int S = p.stages;
  const int nkb = p.nkb, tiles = p.tiles, Kd = p.K;   // in registers: the lambdas below take them by reference
  const long long c = blockIdx.x;
  const long long per_prob = (long long)tiles * nkb;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], DS_NC);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tb_full[b], DS_NC);
      mbar_init(&tb_empty[b], DS_NE);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  span.init();
  for (int i = tid; i < 2 * 16 * DS_RP; i += DS_THREADS) sT[i] = 0.f;
  __syncthreads();
  pdl_launch_dependents();

  // Unit cursor: (live-problem slot li, tile t, k-block kb) of a unit, advanced one unit at a
  // time, so that the loops carry no integer divisions.
  struct Cur {
    int li, t, kb;
  };
  auto cur_at = [&](long long u) {
    Cur r;
    r.li = (int)(u / per_prob);
    const long long rem = u - (long long)r.li * per_prob;
    r.t = (int)(rem / nkb);
    r.kb = (int)(rem - (long long)r.t * nkb);
    return r;
  };
  auto advance = [&](Cur& r) {
    if (++r.kb == nkb) {
      r.kb = 0;
      if (++r.t == tiles) {
        r.t = 0;
        ++r.li;
      }
    }
  };
  auto issue = [&](const Cur& r, int q, int s) {
    mbar_expect_tx(&full[s], (uint32_t)DS_STAGE);
    if (p.bt[q])   // one contiguous 16 KB unit of the tiled copy
      bulk_load(sW + (size_t)s * DS_STAGE, p.bt[q] + ((size_t)r.t * nkb + r.kb) * DS_STAGE, (uint32_t)DS_STAGE,
                &full[s]);
    else
      tma_load_3d(&p.wmap[q], &full[s], sW + (size_t)s * DS_STAGE, r.t * DS_BN, r.kb * (DS_KB / 64));
  };

  // single problem: the partition is known before the wait and the whole ring is issued
  // before it (weights do not depend on the preceding kernel)
  long long U = p.grouped ? 0 : per_prob;
  long long G = U < (long long)gridDim.x ? U : (long long)gridDim.x;
  long long u0 = c < G ? ds_start(c, U, G) : 0, u1 = c < G ? ds_start(c + 1, U, G) : 0;
  int pre = 0;
  if (!p.grouped && warp == 0 && lane == 0) {
    const long long avail = u1 - u0;
    pre = (long long)S > avail ? (int)avail : S;
    Cur r = cur_at(u0);
    for (int g = 0; g < pre; ++g) {
      issue(r, 0, g);
      advance(r);
    }
  }

  DsExitPre xpre;
  if (KIND == EPI_QKV && p.exit_on) ds_exit_prefetch(p, xpre);

  pdl_wait();   // from here on, the preceding kernels' writes are visible
  KT_WAITED();
  span.waited();

  if (KIND == EPI_QKV && p.exit_on) {
    // the previous layer's exit step first: its kept rows are this launch's rows
    if (tid == 0) s_rb[0] = 0;
    ds_exit_stage(p, xpre, sA, s_red, s_M, s_live, &s_nlive, s_tokk, s_bc);
    // the span of the product starts here: the exit step (with the standardised rows it writes)
    // is the previous layer's work, as when it ran as its own kernel before this launch
    span.waited();
  } else {
    // The row counts (device values) and the A operand are read in parallel: every problem's
    // rows start at row 0 (host-checked), so the launch's row bound max_m is staged without
    // waiting for the count (rows past it feed only token columns that are never stored).
    if (warp == 0) {
      // lane q reads problem q's count (all loads at once; MAXG <= 32), the live problems are
      // listed in problem order
      const int q = lane;
      int M = 0;
      if (q < p.n_probs) {
        M = p.rows[q].e();
        if (M > p.max_m) {   // more rows than the launch was sized for
          atomicOr(p.err, ERRW_CONFIG);
          M = p.max_m;
        }
        s_M[q] = M;
        s_rb[q] = 0;
      }
      const unsigned live = __ballot_sync(0xffffffffu, q < p.n_probs && M > 0);
      if (q < p.n_probs && M > 0) s_live[__popc(live & ((1u << q) - 1u))] = q;
      if (lane == 0) s_nlive = __popc(live);
    }
    ds_stage_a(p, sA, p.max_m, s_mu, s_rs, s_red);   // ends with a CTA barrier: the counts are visible
  }
  KT_MARK(1);
  const int nlive = s_nlive;
  if (p.grouped) {
    U = (long long)nlive * per_prob;
    G = U < (long long)gridDim.x ? U : (long long)gridDim.x;
    u0 = c < G ? ds_start(c, U, G) : 0;
    u1 = c < G ? ds_start(c + 1, U, G) : 0;
  }
  if (nlive == 0 || u1 <= u0) {
    // no rows (every token of the step has left), or no units for this CTA: let the copies
    // in flight land, leave
    if (warp == 0 && lane == 0)
      for (int g = 0; g < pre; ++g) ds_wait(&full[g], 0, p.err, DS_TIMEOUT_CYCLES);
    return;
  }
  const int n_units = (int)(u1 - u0);
  const long long gt_first = u0 / nkb, gt_last = (u1 - 1) / nkb;   // this CTA's first / last live-enumerated tile
  const int n_tiles_cta = (int)(gt_last - gt_first + 1);

  if (warp == 0) {
    // ---- producer: refill each slot once its four MMA warps have released it
    if (lane == 0) {
      bool ok = true;
      int issued = pre;
      Cur r = cur_at(u0 + pre);
      int s = pre, n = 0;   // slot and use number of unit g
      if (s == S) {
        s = 0;
        n = 1;
      }
      for (int g = pre; g < n_units && ok; ++g) {
        if (n >= 1) ok = ds_wait(&empty[s], (uint32_t)((n - 1) & 1), p.err, wlim);
        if (ok) {
          issue(r, s_live[r.li], s);
          issued = g + 1;
          advance(r);
          if (++s == S) {
            s = 0;
            ++n;
          }
        }
      }
      // before leaving, every copy this CTA issued has landed (bounded waits; immediate when
      // the MMA warps have taken them)
      for (int h = max(0, issued - S); h < issued; ++h)
        ds_wait(&full[h % S], (uint32_t)((h / S) & 1), p.err, DS_TIMEOUT_CYCLES);
    }
    return;
  }

  if (warp > DS_NC) {
    // ---- epilogue warps: finish each tile the MMA warps hand over, in order
    const int ew = warp - 1 - DS_NC, et = tid - 32 * (1 + DS_NC);   // 0..DS_NE-1, 0..63
    if (KIND == EPI_QKV || KIND == EPI_KV) {
      // each row's position and cache block, looked up once while the first tile streams (every
      // problem of the launch holds the same tokens in the same rows)
      const Epi& e0 = p.epi[s_live[0]];
      int Ms = 0;
      for (int k = 0; k < nlive; ++k) Ms = max(Ms, s_M[s_live[k]]);
      if (et < Ms) {
        const int tok = (KIND == EPI_QKV && p.exit_on) ? s_tokk[et] : e0.row_tok[et];
        const int pos = e0.tok_pos[tok], seq = e0.tok_seq[tok];
        const KVCacheView& cv = e0.cache;
        int blk = -1;
        if (seq >= 0 && seq < cv.max_batch && pos >= 0 && pos < cv.max_blocks_per_seq * cv.block_tokens) {
          blk = cv.block_table[seq * cv.max_blocks_per_seq + pos / cv.block_tokens];
          if (blk < 0 || blk >= cv.n_blocks) blk = -1;
        }
        s_pos[et] = pos;
        s_blk[et] = blk;
      }
      epilogue_sync();
    }
    // one hand-off: the tile's description and sum are in buffer b
    auto process = [&](int b) {
      const int li = s_info[b][0], t = s_info[b][1], whole = s_info[b][2];
      const long long gt = (long long)li * tiles + t;
      const int q = s_live[li];
      const int M = s_M[q], rb = s_rb[q];
      const Epi& e = p.epi[q];
      float* tile = sT + b * 16 * DS_RP;
      if (whole) {
        ds_epilogue<KIND>(e, tile, M, rb, t * DS_BN, p.N, ew, lane, s_pos, s_blk);
        return;
      }
      // shared tile: publish this CTA's partial, count the arrival; the last one finishes it
      const long long slot = 2 * c + (gt == gt_first ? 0 : 1);
      float* mine = p.part + slot * (16 * DS_BN);
      for (int i = et; i < M * DS_BN; i += DS_NE * 32) mine[i] = tile[(i >> 5) * DS_RP + (i & 31)];
      __threadfence();
      epilogue_sync();
      const long long c_first = ds_owner(gt * nkb, U, G), c_last = ds_owner(gt * nkb + nkb - 1, U, G);
      if (et == 0) {
        const int old = atomicAdd(&p.cnt[(long long)q * tiles + t], 1);
        s_last = old == (int)(c_last - c_first);
      }
      epilogue_sync();
      if (!s_last) return;
      __threadfence();
      // the contributors' partials summed in contributor order (each thread at most 8 values)
      float v[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) v[k] = 0.f;
      for (long long cc = c_first; cc <= c_last; ++cc) {
        const long long sl = 2 * cc + (gt == ds_start(cc, U, G) / nkb ? 0 : 1);
        const float* src = p.part + sl * (16 * DS_BN);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int i = et + k * DS_NE * 32;
          if (i < M * DS_BN) v[k] += __ldcg(src + i);
        }
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = et + k * DS_NE * 32;
        if (i < M * DS_BN) tile[(i >> 5) * DS_RP + (i & 31)] = v[k];
      }
      if (et == 0) p.cnt[(long long)q * tiles + t] = 0;
      epilogue_sync();
      ds_epilogue<KIND>(e, tile, M, rb, t * DS_BN, p.N, ew, lane, s_pos, s_blk);
    };
    bool ok = true;
    for (int j = 0; j < n_tiles_cta; ++j) {
      const int b = j & 1;
      bool got = true;
      if (lane == 0 && ok) got = ds_wait(&tb_full[b], (uint32_t)((j >> 1) & 1), p.err, wlim);
      got = __shfl_sync(0xffffffffu, got ? 1 : 0, 0) != 0;
      __syncwarp();     // lane 0's acquire orders the whole warp's reads of the hand-off buffer
      // Both epilogue warps take the same decision: once either has given up, neither reads a
      // hand-off again (its buffer and description may not have been written); they only keep
      // releasing buffers so that the MMA warps finish (outputs undefined, error word set).
      if (lane == 0) s_eok[ew] = (ok && got) ? 1 : 0;
      epilogue_sync();
      ok = s_eok[0] != 0 && s_eok[1] != 0;
      if (ok) process(b);
      epilogue_sync();
      float* tile = sT + b * 16 * DS_RP;
      for (int i = et; i < 16 * DS_RP; i += DS_NE * 32) tile[i] = 0.f;   // zero for the next hand-off
      __syncwarp();
      if (lane == 0) mbar_arrive(&tb_empty[b]);
    }
    return;
  }

  // ---- MMA warps: warp cw = (mb, kh): features mb*16.., 64-k chunks kh, kh + 2 of a unit
  const int cw = warp - 1, mb = cw & 1, kh = cw >> 1;
  const int wrow = mb * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
  const uint32_t w_base = smem_u32(sW) + kh * DS_CHUNK + wrow * 128;
  const int wx = wrow & 7, wu = (lane >> 4) & 1;
  const int ap = p.apitch;
  const uint32_t a_base = smem_u32(sA) + ((lane & 7) + ((lane >> 4) & 1) * 8) * ap * 2 + ((lane >> 3) & 1) * 16 +
                          kh * 128;
  const int bg = lane >> 2;
  const uint32_t b_base = smem_u32(sA) + (bg * ap + kh * 64 + (lane & 3) * 2) * 2;

  // one accumulator set per k16 step of a 64-k chunk: four independent MMA chains per warp
  float acc[4][MB][4];
  auto zero_acc = [&]() {
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
      for (int t = 0; t < MB; ++t) acc[k][t][0] = acc[k][t][1] = acc[k][t][2] = acc[k][t][3] = 0.f;
  };
  zero_acc();
  Cur r = cur_at(u0);

  // Every lane waits for each slot and one vote makes the decision warp-uniform (the fragment
  // loads and MMAs below are .aligned).  A warp whose wait gives up stops waiting, computing and
  // releasing slots (a slot it has not seen land must not be refilled: the producer's own
  // bounded wait then ends the stream and it drains its copies), but still hands over every
  // tile, so the epilogue warps and the CTA complete (the error word is set).
  bool ok = true;
  bool seg_whole_start = r.kb == 0;   // the current tile's segment began at its first k-block
  int Mq = s_M[s_live[r.li]];
  int s = 0, n = 0;                   // slot and use number of unit g
  int j = 0;                          // tile hand-offs so far
  for (int g = 0; g < n_units; ++g) {
    if (ok)   // every lane polls; one vote makes the outcome warp-uniform (.aligned MMAs below)
      ok = __all_sync(0xffffffffu, ds_wait(&full[s], (uint32_t)(n & 1), p.err, wlim)) != 0;
    const int kb = r.kb;
    const int nch = ok ? min(DS_KB, Kd - kb * DS_KB) >> 6 : 0;
    const uint32_t sbase = w_base + s * DS_STAGE;
    for (int q = 0; 2 * q + kh < nch; ++q) {
      const uint32_t wa = sbase + q * (2 * DS_CHUNK);
      const int kk0 = kb * DS_KB + q * 128;
      const uint32_t aa = a_base + kk0 * 2;
      const uint32_t ab = b_base + kk0 * 2;
      // every fragment of the chunk first, then four independent MMAs
      uint32_t a[4][4];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) ldsm_x4(a[kk], wa + (((kk * 2 + wu) ^ wx) << 4));
      if (MB == 2) {
        uint32_t bb[4][4];
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) ldsm_x4(bb[kk], aa + kk * 32);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          mma_bf16(acc[kk][0], a[kk], bb[kk][0], bb[kk][1]);
          mma_bf16(acc[kk][MB - 1], a[kk], bb[kk][2], bb[kk][3]);
        }
      } else {
        uint32_t b0[4], b1[4];
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          b0[kk] = b1[kk] = 0u;
          if (bg < Mq) {
            b0[kk] = ld_shared_u32(ab + kk * 32);
            b1[kk] = ld_shared_u32(ab + kk * 32 + 16);
          }
        }
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) mma_bf16(acc[kk][0], a[kk], b0[kk], b1[kk]);
      }
    }
    __syncwarp();
    if (lane == 0 && ok) mbar_arrive(&empty[s]);
    const bool last = g == n_units - 1;
    if (kb == nkb - 1 || last) {
      // hand the tile over: wait until the buffer is free, add this warp's k half into it
      // (exactly two additions per element onto zero, so the sum does not depend on their
      // order), signal the epilogue warps
      const int b = j & 1;
      if (j >= 2) {
        bool free_ok = true;
        if (lane == 0) free_ok = ds_wait(&tb_empty[b], (uint32_t)(((j >> 1) - 1) & 1), p.err, wlim);
        free_ok = __shfl_sync(0xffffffffu, free_ok ? 1 : 0, 0) != 0;
        __syncwarp();
        ok = ok && free_ok;
      }
      if (cw == 0 && lane == 0) {
        s_info[b][0] = r.li;
        s_info[b][1] = r.t;
        s_info[b][2] = (seg_whole_start && kb == nkb - 1) ? 1 : 0;
      }
      float* tile = sT + b * 16 * DS_RP;
      const int gq = lane >> 2, t4 = lane & 3;
#pragma unroll
      for (int t2 = 0; t2 < MB; ++t2) {
        float a4[4];
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) a4[jj] = (acc[0][t2][jj] + acc[1][t2][jj]) + (acc[2][t2][jj] + acc[3][t2][jj]);
        const int tk = t2 * 8 + 2 * t4, fc = mb * 16 + gq;
        atomicAdd(&tile[tk * DS_RP + fc], a4[0]);
        atomicAdd(&tile[(tk + 1) * DS_RP + fc], a4[1]);
        atomicAdd(&tile[tk * DS_RP + fc + 8], a4[2]);
        atomicAdd(&tile[(tk + 1) * DS_RP + fc + 8], a4[3]);
      }
      zero_acc();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tb_full[b]);
      ++j;
      seg_whole_start = true;
    }
    advance(r);
    if (++s == S) {
      s = 0;
      ++n;
    }
    if (r.kb == 0 && !last) Mq = s_M[s_live[r.li]];
  }
  KT_MARK(6);
}

int g_ds_sms = 0;
int g_ds_sm_smem = 0;   // shared memory per SM (bytes)

template <int MB, int KIND, int MAXG>
cudaError_t ds_launch(cudaStream_t st, const DsParams<MAXG>& prm, int grid, size_t smem) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(gemm_stream_kernel<MB, KIND, MAXG>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, DS_SMEM_LIMIT);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(DS_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<MB, KIND, MAXG>, prm);
}

template <int MB, int MAXG>
cudaError_t ds_launch_kind(cudaStream_t st, const DsParams<MAXG>& prm, int grid, size_t smem) {
  switch (prm.epi[0].kind) {
    case EPI_F32: return ds_launch<MB, EPI_F32, MAXG>(st, prm, grid, smem);
    case EPI_ACT: return ds_launch<MB, EPI_ACT, MAXG>(st, prm, grid, smem);
    case EPI_RESID: return ds_launch<MB, EPI_RESID, MAXG>(st, prm, grid, smem);
    case EPI_SWIGLU: return ds_launch<MB, EPI_SWIGLU, MAXG>(st, prm, grid, smem);
    case EPI_QKV: return ds_launch<MB, EPI_QKV, MAXG>(st, prm, grid, smem);
    default: return ds_launch<MB, EPI_KV, MAXG>(st, prm, grid, smem);
  }
}

// Host plan shared by the single and the grouped launch: checks, tile counts, shared-memory
// layout and ring depth.  False when the stream-K path does not take the shape.
template <int MAXG>
bool ds_plan(const GemmProblem& q, int n_probs, int max_rows, const DgNorm* norm, const DsWork& ws, unsigned* err,
             DsParams<MAXG>& prm, int& grid, size_t& smem, int& mb) {
  if (!ws.part || !ws.cnt) return false;
  if (max_rows <= 0 || max_rows > 16 || q.N <= 0 || q.K <= 0 || q.K % 64) return false;
  if (q.ldb % 8 || ((uintptr_t)q.B & 15)) return false;
  if (!norm && (q.lda % 8 || ((uintptr_t)q.A & 15))) return false;
  if (norm && (!norm->X || norm->ldx % 4 || ((uintptr_t)norm->X & 15) || q.K % 4)) return false;
  if ((q.epi.kind == EPI_QKV || q.epi.kind == EPI_KV || q.epi.kind == EPI_SWIGLU) && q.N % 32) return false;
  if (q.epi.tile_stats && (q.epi.kind != EPI_RESID || q.N % DS_BN)) return false;
  if (q.epi.kind < EPI_F32 || q.epi.kind > EPI_KV) return false;
  if ((long long)q.N * q.K * 2 * n_probs < DS_MIN_STREAM_BYTES) return false;
  // narrow single problems (N < DS_MIN_N: every CTA would hold less than about two tiles and
  // end on a shared tile's fix-up) stream faster on the cluster K-split kernel, whose partial
  // sums meet in distributed shared memory (measured at the Llama-7B O and down projections)
  if (n_probs == 1 && q.N < DS_MIN_N) return false;
  if (q.rows.begin) return false;   // rows start at 0: the operand is staged before the count is read
  if (norm && q.K > DS_XV * 4 * DS_THREADS) return false;
  if (!g_ds_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_ds_sms, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&g_ds_sm_smem, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
    if (g_ds_sms <= 0) g_ds_sms = 1;
  }
  grid = g_ds_sms;
  if (grid > ws.part_ctas) return false;
  const int tiles = cdiv(q.N, DS_BN);
  if ((long long)tiles * n_probs > ws.cnt_cap) return false;
  mb = max_rows > 8 ? 2 : 1;
  const int arows = mb == 2 ? 16 : max_rows;
  const int apitch = q.K + 8;   // 16-byte shift per row: conflict-free fragment loads
  const int a_bytes = ((arows * apitch * 2) + 127) & ~127;
  const int p_bytes = 2 * 16 * DS_RP * 4;   // the two tile hand-off buffers
  const int fixed = 1024 + a_bytes + p_bytes;
  const int STATIC = 2 * DS_MAX_STAGES * 8 + 32 + 128 + DS_WARPS * 64 + 3 * MAXG * 4 + 16 + 128 + 24 + 64;
  const int stages = std::min(DS_RING_STAGES, (DS_SMEM_LIMIT - STATIC - fixed) / DS_STAGE);
  if (stages < 2) return false;
  memset(&prm, 0, sizeof prm);
  prm.n_probs = n_probs;
  prm.tiles = tiles;
  prm.nkb = cdiv(q.K, DS_KB);
  prm.N = q.N;
  prm.K = q.K;
  prm.stages = stages;
  prm.max_m = max_rows;
  prm.arows = arows;
  prm.apitch = apitch;
  prm.off_a = stages * DS_STAGE;
  prm.off_p = prm.off_a + a_bytes;
  prm.A = (const bf16*)q.A;
  prm.lda = q.lda;
  prm.X = norm ? norm->X : nullptr;
  prm.ldx = norm ? norm->ldx : 0;
  prm.in_rows = norm ? norm->in_rows : nullptr;
  prm.norm_mode = norm ? norm->mode : NORM_COPY;
  prm.eps = norm ? norm->eps : 0.f;
  prm.fused_norm = norm != nullptr;
  prm.stat_mode = !norm ? DS_STATS_HERE
                  : norm->row_stats ? DS_STATS_ROWS
                  : (norm->tile_stats && q.K % 32 == 0) ? DS_STATS_TILES
                                                         : DS_STATS_HERE;
  prm.row_stats = norm ? norm->row_stats : nullptr;
  prm.tile_stats = norm ? norm->tile_stats : nullptr;
  prm.n_stiles = q.K / 32;
  prm.part = ws.part;
  prm.cnt = ws.cnt;
  prm.err = err;
  prm.span = g_span;
  smem = (size_t)prm.off_p + p_bytes + 1024;
  smem = std::max(smem, (size_t)g_ds_sm_smem / 2 + 1024);   // no second CTA of this kernel on the SM
  return smem <= (size_t)DS_SMEM_LIMIT;
}

// The problem's tile-contiguous copy when its layout matches the launch (k-blocks per tile,
// 16-byte alignment), else NULL (the tensor map on B is used).
const uint8_t* ds_tiled(const GemmProblem& q, int nkb) {
  if (!q.Bt || q.bt_nkb != nkb || ((uintptr_t)q.Bt & 15)) return nullptr;
  return (const uint8_t*)q.Bt;
}

}  // namespace

size_t stream_gemm_part_bytes(int sms) { return (size_t)2 * sms * 16 * DS_BN * sizeof(float); }

int stream_gemm(cudaStream_t st, const GemmProblem& q, int max_rows, const DgNorm* norm, const DsWork& ws,
                unsigned* err) {
  thread_local DsParams<1> prm;   // one per host thread
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!ds_plan(q, 1, max_rows, norm, ws, err, prm, grid, smem, mb)) return -1;
  prm.bt[0] = ds_tiled(q, prm.nkb);   // the tensor map is read only without the tiled copy
  if (!prm.bt[0] && !tc_encode_weight_3d(&prm.wmap[0], q.B, q.K, q.N, (size_t)q.ldb * 2, DS_BN, DS_KB / 64))
    return -1;
  prm.grouped = 0;
  prm.rows[0] = q.rows;
  prm.epi[0] = q.epi;
  const cudaError_t e = mb == 2 ? ds_launch_kind<2, 1>(st, prm, grid, smem) : ds_launch_kind<1, 1>(st, prm, grid, smem);
  return e == cudaSuccess ? 1 : -1;
}

int stream_gemm_exit(cudaStream_t st, const GemmProblem& q, int max_rows, const DsExit& ex, const DsWork& ws,
                     unsigned* err) {
  if (q.epi.kind != EPI_QKV || max_rows < 1 || max_rows > DS_EXIT_MAX_ROWS) return -1;
  if (q.K % 4 || q.K / 4 > DS_XV * DS_THREADS || ex.layer < 1 || ex.layer >= ex.n_layers) return -1;
  if (ex.metric != EXIT_GLOBAL) return -1;   // the local rules also need s_{i-1}'s sums
  if (!ex.Xin || !ex.Xout || !ex.I || !ex.Xnext || !ex.Inext || !ex.hsm_s || !ex.hsm_prev || !ex.hsm_I || !ex.ctr ||
      !ex.row_tok || !ex.row_tok_next || !ex.delta || !ex.exit_tok)
    return -1;
  const uintptr_t al = (uintptr_t)ex.Xin | (uintptr_t)ex.Xout | (uintptr_t)ex.I | (uintptr_t)ex.Xnext |
                       (uintptr_t)ex.Inext | (uintptr_t)ex.hsm_s | (uintptr_t)ex.hsm_prev | (uintptr_t)ex.hsm_I;
  if (al & 15) return -1;
  thread_local DsParams<1> prm;   // one per host thread
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!ds_plan(q, 1, max_rows, nullptr, ws, err, prm, grid, smem, mb)) return -1;
  prm.bt[0] = ds_tiled(q, prm.nkb);
  if (!prm.bt[0] && !tc_encode_weight_3d(&prm.wmap[0], q.B, q.K, q.N, (size_t)q.ldb * 2, DS_BN, DS_KB / 64))
    return -1;
  prm.grouped = 0;
  prm.rows[0] = q.rows;
  prm.epi[0] = q.epi;
  prm.exit_on = 1;
  prm.ex = ex;
  const cudaError_t e = mb == 2 ? ds_launch<2, EPI_QKV, 1>(st, prm, grid, smem) : ds_launch<1, EPI_QKV, 1>(st, prm, grid, smem);
  return e == cudaSuccess ? 1 : -1;
}

int stream_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n, int max_rows, const DsWork& ws,
                        unsigned* err) {
  if (n < 1 || n > DS_MAXG) return -1;
  const GemmProblem& q0 = probs[0];
  for (int i = 0; i < n; ++i) {
    const GemmProblem& q = probs[i];
    if (q.epi.kind != EPI_KV || q.A != q0.A || q.lda != q0.lda || q.N != q0.N || q.K != q0.K || q.ldb != q0.ldb ||
        q.rows.begin != nullptr || q.epi.tile_stats)
      return -1;
  }
  thread_local DsParams<DS_MAXG> prm;
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!ds_plan(q0, n, max_rows, nullptr, ws, err, prm, grid, smem, mb)) return -1;
  for (int i = 0; i < n; ++i) {
    prm.bt[i] = ds_tiled(probs[i], prm.nkb);   // the tensor map is read only without the tiled copy
    if (!prm.bt[i] && (((uintptr_t)probs[i].B & 15) ||
                       !tc_encode_weight_3d(&prm.wmap[i], probs[i].B, q0.K, q0.N, (size_t)q0.ldb * 2, DS_BN,
                                            DS_KB / 64)))
      return -1;
    prm.rows[i] = probs[i].rows;
    prm.epi[i] = probs[i].epi;
  }
  prm.grouped = 1;
  const cudaError_t e = mb == 2 ? ds_launch<2, EPI_KV, DS_MAXG>(st, prm, grid, smem)
                                : ds_launch<1, EPI_KV, DS_MAXG>(st, prm, grid, smem);
  return e == cudaSuccess ? 1 : -1;
}

ADEPT_WAIT_LIMIT_SETTER(ds)

}  // namespace adept

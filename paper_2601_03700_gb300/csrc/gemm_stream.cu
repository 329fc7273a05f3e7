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
//    so the first slots are issued before the programmatic-dependent-launch wait.  The CTA
//    is sized (about 112 KB of shared memory) so that the next launch's CTA fits beside it
//    on the SM and its first copies overlap this launch's tail.
//  * A operand: after the wait the launch's token rows (all of K) are staged once in shared
//    memory, copied (bf16) or standardised from the fp32 residual stream with row statistics
//    computed here or handed over by the producer of the rows.
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

#include <cuda.h>

#include <algorithm>
#include <cstring>

namespace adept {
namespace {

constexpr int DS_BN = 32;                         // output features per tile
constexpr int DS_KB = 256;                        // k per unit
constexpr int DS_CHUNK = DS_BN * 128;             // one [32 rows][64 k] 128-byte-swizzled chunk
constexpr int DS_STAGE = DS_BN * DS_KB * 2;       // 16 KB per unit
constexpr int DS_NC = 4;                          // consumer warps
constexpr int DS_THREADS = 32 * (DS_NC + 1);      // + the producer warp
constexpr int DS_MAX_STAGES = 12;
constexpr int DS_PRE = 3;                         // units issued before the dependency wait
constexpr int DS_RP = DS_BN + 1;                  // floats per token row of a partial tile
constexpr int DS_MAXG = 32;
constexpr int DS_COHOST_SMEM = 113 * 1024;        // two launches' CTAs fit on one SM (228 KB, 1 KB each reserved)
constexpr int DS_SMEM_LIMIT = 200 * 1024;
constexpr long long DS_TIMEOUT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz
constexpr long long DS_MIN_STREAM_BYTES = 8ll << 20;    // below: the cluster K-split kernel
enum : int { DS_STATS_HERE = 0, DS_STATS_ROWS = 1, DS_STATS_TILES = 2 };

template <int MAXG>
struct DsParams {
  CUtensorMap wmap[MAXG];   // W as {64, N, K/64}, box {64, 32, 4}, 128-byte swizzle
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
// Barrier of the consumer warps only (the producer keeps streaming meanwhile).
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(DS_NC * 32) : "memory"); }

// Stream-K partition of U units over G CTAs: CTA c takes [start(c), start(c + 1)).
__device__ __forceinline__ long long ds_start(long long c, long long U, long long G) { return c * U / G; }
// The CTA whose range holds unit u (the last CTA c with start(c) <= u).
__device__ __forceinline__ long long ds_owner(long long u, long long U, long long G) {
  return ((u + 1) * G + U - 1) / U - 1;
}

// Fused epilogue of one tile, element-parallel over the consumer warps: warp cw takes rows
// cw, cw + DS_NC, ..., lane = feature.
template <int KIND>
__device__ __forceinline__ void ds_epilogue(const Epi& e, const float* sS, int M, int rb, int f0, int N, int cw,
                                            int lane, const int* s_pos, const int* s_blk) {
  for (int row = cw; row < M; row += DS_NC) {
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

// Stages rows [rb, rb + M) of the A operand into sA (bf16, pitch apitch; all K), rows
// M..arows-1 zero.  All threads of the CTA take part.
template <int MAXG>
__device__ void ds_stage_a(const DsParams<MAXG>& p, bf16* sA, int rb, int M, float* s_mu, float* s_rs,
                           float (*s_red)[16]) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, K = p.K, ap = p.apitch;
  for (int i = tid; i < (p.arows - M) * (ap >> 3); i += DS_THREADS) {   // zero rows past M
    const int r = M + i / (ap >> 3), c = i % (ap >> 3);
    *reinterpret_cast<uint4*>(sA + (size_t)r * ap + c * 8) = make_uint4(0, 0, 0, 0);
  }
  if (!p.fused_norm) {
    const int cpr = K >> 3;
    for (int i = tid; i < M * cpr; i += DS_THREADS) {
      const int r = i / cpr, c = i - r * cpr;
      cp_async16(sA + (size_t)r * ap + c * 8, p.A + (size_t)(rb + r) * p.lda + c * 8);
    }
    cp_async_wait_all();
    __syncthreads();
    return;
  }
  // row statistics (mu, rstd) of the fp32 source rows
  const float* xr[16];
#pragma unroll
  for (int r = 0; r < 16; ++r) xr[r] = p.X + (size_t)(r < M ? (p.in_rows ? p.in_rows[rb + r] : rb + r) : 0) * p.ldx;
  if (p.stat_mode == DS_STATS_ROWS) {
    if (tid < M) {
      const float2 s = p.row_stats[rb + tid];
      s_mu[tid] = s.x;
      s_rs[tid] = s.y;
    }
  } else if (p.stat_mode == DS_STATS_TILES) {
    // the row's moments from the producer's 32-column (mean, M2) tiles, about the first
    // tile's mean c: S1 = sum 32 (m_t - c), S2 = sum M2_t + 32 (m_t - c)^2
    for (int r = warp; r < M; r += DS_NC + 1) {
      const float2* ts = p.tile_stats + (size_t)(rb + r) * p.n_stiles;
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
    // two passes over the rows (L2-resident): mean, then the centred second moment
    auto row_sums = [&](auto term, float* out) {
      float part[16];
#pragma unroll
      for (int r = 0; r < 16; ++r) part[r] = 0.f;
      for (int d = tid * 4; d < K; d += DS_THREADS * 4) {
#pragma unroll
        for (int r = 0; r < 16; ++r)
          if (r < M) {
            const float4 x = *reinterpret_cast<const float4*>(xr[r] + d);
            part[r] += term(r, x.x) + term(r, x.y) + term(r, x.z) + term(r, x.w);
          }
      }
#pragma unroll
      for (int r = 0; r < 16; ++r) {
        const float v = warp_sum(part[r]);
        if (lane == 0) s_red[warp][r] = v;
      }
      __syncthreads();
      if (tid < M) {
        float t = 0.f;
        for (int w = 0; w < DS_NC + 1; ++w) t += s_red[w][tid];
        out[tid] = t / K;
      }
      __syncthreads();
    };
    if (tid < 16) {
      s_mu[tid] = 0.f;
      s_rs[tid] = 1.f;
    }
    __syncthreads();
    if (p.norm_mode == NORM_LN) row_sums([](int, float x) { return x; }, s_mu);
    if (p.norm_mode != NORM_COPY) {
      row_sums([&](int r, float x) { const float c = x - s_mu[r]; return c * c; }, s_rs);
      if (tid < M) s_rs[tid] = rsqrtf(s_rs[tid] + p.eps);
    }
  }
  __syncthreads();
  for (int i = tid; i < M * (K >> 2); i += DS_THREADS) {
    const int r = i / (K >> 2), v4 = i - r * (K >> 2);
    const float4 x = *reinterpret_cast<const float4*>(xr[r] + v4 * 4);
    const float mu = s_mu[r], rs = s_rs[r];
    const __nv_bfloat162 lo = __floats2bfloat162_rn((x.x - mu) * rs, (x.y - mu) * rs);
    const __nv_bfloat162 hi = __floats2bfloat162_rn((x.z - mu) * rs, (x.w - mu) * rs);
    uint2 u;
    u.x = *reinterpret_cast<const uint32_t*>(&lo);
    u.y = *reinterpret_cast<const uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(sA + (size_t)r * ap + v4 * 4) = u;
  }
  __syncthreads();
}

// MB: 8-token blocks of the A operand (1: M <= 8, 2: M <= 16); KIND: the epilogue kind.
template <int MB, int KIND, int MAXG>
__global__ void __launch_bounds__(DS_THREADS, 1) gemm_stream_kernel(const __grid_constant__ DsParams<MAXG> p) {
  KT_BEGIN();
  extern __shared__ __align__(128) uint8_t ds_smem_raw[];
  __shared__ __align__(8) uint64_t full[DS_MAX_STAGES];
  __shared__ __align__(8) uint64_t empty[DS_MAX_STAGES];
  __shared__ float s_mu[16], s_rs[16];
  __shared__ float s_red[DS_NC + 1][16];
  __shared__ int s_live[MAXG];     // problems with rows, in order
  __shared__ int s_M[MAXG], s_rb[MAXG];
  __shared__ int s_nlive, s_last;
  __shared__ int s_pos[16], s_blk[16];   // cache epilogues: each row's position and cache block

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint8_t* smem = ds_smem_raw + ((1024 - (smem_u32(ds_smem_raw) & 1023)) & 1023);
  uint8_t* sW = smem;                                           // [S][4 chunks][32 rows][128 B], swizzled
  bf16* sA = reinterpret_cast<bf16*>(smem + p.off_a);           // [arows][apitch]
  float* sP = reinterpret_cast<float*>(smem + p.off_p);         // [2][16][DS_RP] k halves, then [16][DS_RP] sum
  float* sS = sP + 2 * 16 * DS_RP;
  const int S = p.stages;
  const long long c = blockIdx.x;
  const long long per_prob = (long long)p.tiles * p.nkb;
  // the units are shared by G = min(grid, units) CTAs, so that every sharing CTA has at
  // least one unit (a tile's contributors are then exactly the CTAs between its first and
  // its last unit's owners)

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], DS_NC);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
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
    r.t = (int)(rem / p.nkb);
    r.kb = (int)(rem - (long long)r.t * p.nkb);
    return r;
  };
  auto advance = [&](Cur& r) {
    if (++r.kb == p.nkb) {
      r.kb = 0;
      if (++r.t == p.tiles) {
        r.t = 0;
        ++r.li;
      }
    }
  };
  auto issue = [&](const Cur& r, int q, int s) {
    mbar_expect_tx(&full[s], (uint32_t)DS_STAGE);
    tma_load_3d(&p.wmap[q], &full[s], sW + (size_t)s * DS_STAGE, r.t * DS_BN, r.kb * (DS_KB / 64));
  };

  // single problem: the partition is known before the wait; its first units are issued
  // before it (weights do not depend on the preceding kernel)
  long long U = p.grouped ? 0 : per_prob;
  long long G = U < (long long)gridDim.x ? U : (long long)gridDim.x;
  long long u0 = c < G ? ds_start(c, U, G) : 0, u1 = c < G ? ds_start(c + 1, U, G) : 0;
  int pre = 0;
  if (!p.grouped && warp == 0 && lane == 0) {
    const long long avail = u1 - u0;
    pre = S < DS_PRE ? S : DS_PRE;
    if ((long long)pre > avail) pre = (int)avail;
    Cur r = cur_at(u0);
    for (int g = 0; g < pre; ++g) {
      issue(r, 0, g);
      advance(r);
    }
  }

  pdl_wait();   // from here on, the preceding kernels' writes are visible
  KT_WAITED();

  if (tid == 0) {
    int n = 0;
    for (int q = 0; q < p.n_probs; ++q) {
      const int b = p.rows[q].b();
      int M = p.rows[q].e() - b;
      if (M > p.max_m) {   // more rows than the launch was sized for
        atomicOr(p.err, ERRW_CONFIG);
        M = p.max_m;
      }
      s_M[q] = M;
      s_rb[q] = b;
      if (M > 0) s_live[n++] = q;
    }
    s_nlive = n;
  }
  __syncthreads();
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

  // A operand: the rows of the launch (grouped: every problem's rows are a prefix of one
  // shared range starting at the first live problem's begin)
  int Ms = 0;
  for (int k = 0; k < nlive; ++k) Ms = max(Ms, s_M[s_live[k]]);
  const int rb0 = s_rb[s_live[0]];
  if (KIND == EPI_QKV || KIND == EPI_KV) {
    // each row's position and cache block, looked up once (every problem of the launch holds
    // the same tokens in the same rows)
    const Epi& e0 = p.epi[s_live[0]];
    if (tid < Ms) {
      const int tok = e0.row_tok[rb0 + tid];
      const int pos = e0.tok_pos[tok], seq = e0.tok_seq[tok];
      const KVCacheView& cv = e0.cache;
      int blk = -1;
      if (seq >= 0 && seq < cv.max_batch && pos >= 0 && pos < cv.max_blocks_per_seq * cv.block_tokens) {
        blk = cv.block_table[seq * cv.max_blocks_per_seq + pos / cv.block_tokens];
        if (blk < 0 || blk >= cv.n_blocks) blk = -1;
      }
      s_pos[tid] = pos;
      s_blk[tid] = blk;
    }
  }
  ds_stage_a(p, sA, rb0, Ms, s_mu, s_rs, s_red);
  KT_MARK(1);

  if (warp == 0) {
    // ---- producer: refill each slot once its four consumer warps have released it
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
        if (n >= 1) ok = ds_wait(&empty[s], (uint32_t)((n - 1) & 1), p.err, wait_limit());
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
      // the consumers have taken them)
      for (int h = max(0, issued - S); h < issued; ++h)
        ds_wait(&full[h % S], (uint32_t)((h / S) & 1), p.err, DS_TIMEOUT_CYCLES);
    }
    return;
  }

  // ---- consumers: warp cw = (mb, kh): features mb*16.., 64-k chunks kh, kh + 2 of a unit
  const int cw = warp - 1, mb = cw & 1, kh = cw >> 1;
  const int wrow = mb * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
  const uint32_t w_base = smem_u32(sW) + kh * DS_CHUNK + wrow * 128;
  const int wx = wrow & 7, wu = (lane >> 4) & 1;
  const int ap = p.apitch;
  const uint32_t a_base = smem_u32(sA) + ((lane & 7) + ((lane >> 4) & 1) * 8) * ap * 2 + ((lane >> 3) & 1) * 16 +
                          kh * 128;
  const int bg = lane >> 2;
  const uint32_t b_base = smem_u32(sA) + (bg * ap + kh * 64 + (lane & 3) * 2) * 2;
  const int ct = tid - 32;   // 0..127 among the consumers

  float acc[MB][4];
  auto zero_acc = [&]() {
#pragma unroll
    for (int t = 0; t < MB; ++t) acc[t][0] = acc[t][1] = acc[t][2] = acc[t][3] = 0.f;
  };
  zero_acc();
  Cur r = cur_at(u0);
  const long long gt_first = (long long)r.li * p.tiles + r.t;   // this CTA's first (live-enumerated) tile

  // the tile (li, t) ends here; whole: this CTA covered all of its k-blocks
  auto finish_tile = [&](int li, int t, bool whole) {
    const long long gt = (long long)li * p.tiles + t;
    const int q = s_live[li];
    const int M = s_M[q], rb = s_rb[q];
    const Epi& e = p.epi[q];
    // partial tile [token][feature] of this warp into its k half, then the sum of halves
    {
      float* part = sP + kh * 16 * DS_RP;
      const int gq = lane >> 2, t4 = lane & 3;
#pragma unroll
      for (int t2 = 0; t2 < MB; ++t2) {
        const int tk = t2 * 8 + 2 * t4, fc = mb * 16 + gq;
        part[tk * DS_RP + fc] = acc[t2][0];
        part[(tk + 1) * DS_RP + fc] = acc[t2][1];
        part[tk * DS_RP + fc + 8] = acc[t2][2];
        part[(tk + 1) * DS_RP + fc + 8] = acc[t2][3];
      }
    }
    zero_acc();
    consumers_sync();
    for (int i = ct; i < M * DS_BN; i += DS_NC * 32) {
      const int j = (i >> 5) * DS_RP + (i & 31);
      sS[j] = sP[j] + sP[16 * DS_RP + j];
    }
    consumers_sync();
    if (!whole) {
      // shared tile: publish this CTA's partial, count the arrival; the last one finishes it
      const long long slot = 2 * c + (gt == gt_first ? 0 : 1);
      float* mine = p.part + slot * (16 * DS_BN);
      for (int i = ct; i < M * DS_BN; i += DS_NC * 32) mine[i] = sS[(i >> 5) * DS_RP + (i & 31)];
      __threadfence();
      consumers_sync();
      const long long c_first = ds_owner(gt * p.nkb, U, G), c_last = ds_owner(gt * p.nkb + p.nkb - 1, U, G);
      if (ct == 0) {
        const int old = atomicAdd(&p.cnt[(long long)q * p.tiles + t], 1);
        s_last = old == (int)(c_last - c_first);
      }
      consumers_sync();
      if (!s_last) return;
      __threadfence();
      // the contributors' partials summed in contributor order (each thread at most 4 values)
      float v[4] = {0.f, 0.f, 0.f, 0.f};
      for (long long cc = c_first; cc <= c_last; ++cc) {
        const long long sl = 2 * cc + (gt == ds_start(cc, U, G) / p.nkb ? 0 : 1);
        const float* src = p.part + sl * (16 * DS_BN);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int i = ct + k * DS_NC * 32;
          if (i < M * DS_BN) v[k] += __ldcg(src + i);
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = ct + k * DS_NC * 32;
        if (i < M * DS_BN) sS[(i >> 5) * DS_RP + (i & 31)] = v[k];
      }
      if (ct == 0) p.cnt[(long long)q * p.tiles + t] = 0;
      consumers_sync();
    }
    ds_epilogue<KIND>(e, sS, M, rb, t * DS_BN, p.N, cw, lane, s_pos, s_blk);
    consumers_sync();   // sP / sS are rewritten by the next tile
  };

  // A warp whose wait gives up stops waiting and computing but still releases its slots and
  // takes part in every consumer barrier, so the CTA always completes (the error word is set).
  bool ok = true;
  bool seg_whole_start = r.kb == 0;   // the current tile's segment began at its first k-block
  int Mq = s_M[s_live[r.li]];
  int s = 0, n = 0;                   // slot and use number of unit g
  for (int g = 0; g < n_units; ++g) {
    if (ok) ok = ds_wait(&full[s], (uint32_t)(n & 1), p.err, wait_limit());
    const int kb = r.kb;
    const int nch = ok ? min(DS_KB, p.K - kb * DS_KB) >> 6 : 0;
    const uint32_t sbase = w_base + s * DS_STAGE;
    for (int q = 0; 2 * q + kh < nch; ++q) {
      const uint32_t wa = sbase + q * (2 * DS_CHUNK);
      const int kk0 = kb * DS_KB + q * 128;
      const uint32_t aa = a_base + kk0 * 2;
      const uint32_t ab = b_base + kk0 * 2;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t a[4];
        ldsm_x4(a, wa + (((kk * 2 + wu) ^ wx) << 4));
        if (MB == 2) {
          uint32_t b[4];
          ldsm_x4(b, aa + kk * 32);
          mma_bf16(acc[0], a, b[0], b[1]);
          mma_bf16(acc[MB - 1], a, b[2], b[3]);
        } else {
          uint32_t b0 = 0u, b1 = 0u;
          if (bg < Mq) {
            b0 = ld_shared_u32(ab + kk * 32);
            b1 = ld_shared_u32(ab + kk * 32 + 16);
          }
          mma_bf16(acc[0], a, b0, b1);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
    const bool last = g == n_units - 1;
    // tile boundary or the end of the range: finish the tile
    if (kb == p.nkb - 1 || last) {
      finish_tile(r.li, r.t, seg_whole_start && kb == p.nkb - 1);
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
  if (!g_ds_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_ds_sms, cudaDevAttrMultiProcessorCount, dev);
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
  const int p_bytes = 3 * 16 * DS_RP * 4;
  const int fixed = 1024 + a_bytes + p_bytes;
  const int STATIC = 2 * DS_MAX_STAGES * 8 + 64 * 4 + (DS_NC + 1) * 64 + 3 * MAXG * 4 + 64 + 128;
  int stages = (DS_COHOST_SMEM - STATIC - fixed) / DS_STAGE;
  if (stages < 4) stages = (DS_SMEM_LIMIT - STATIC - fixed) / DS_STAGE;
  if (stages < 2) return false;
  stages = std::min(stages, DS_MAX_STAGES);
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
  smem = (size_t)prm.off_p + p_bytes + 1024;
  return smem <= (size_t)DS_SMEM_LIMIT;
}

}  // namespace

size_t stream_gemm_part_bytes(int sms) { return (size_t)2 * sms * 16 * DS_BN * sizeof(float); }

int stream_gemm(cudaStream_t st, const GemmProblem& q, int max_rows, const DgNorm* norm, const DsWork& ws,
                unsigned* err) {
  thread_local DsParams<1> prm;   // one per host thread
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!ds_plan(q, 1, max_rows, norm, ws, err, prm, grid, smem, mb)) return -1;
  if (!tc_encode_weight_3d(&prm.wmap[0], q.B, q.K, q.N, (size_t)q.ldb * 2, DS_BN, DS_KB / 64)) return -1;
  prm.grouped = 0;
  prm.rows[0] = q.rows;
  prm.epi[0] = q.epi;
  const cudaError_t e = mb == 2 ? ds_launch_kind<2, 1>(st, prm, grid, smem) : ds_launch_kind<1, 1>(st, prm, grid, smem);
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
    if (((uintptr_t)probs[i].B & 15) ||
        !tc_encode_weight_3d(&prm.wmap[i], probs[i].B, q0.K, q0.N, (size_t)q0.ldb * 2, DS_BN, DS_KB / 64))
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

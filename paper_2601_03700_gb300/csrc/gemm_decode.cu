// Generation-step GEMM for sm_103a: C[M, N] = A[M, K] * W[N, K]^T with M <= 16 token rows.
// Such a pass multiplies every weight once (8 flops per weight byte at M = 8, far below
// the tensor-core ridge), so it is a stream over W and the design maximises the weight
// bytes in flight and hides start-up latency; the MMA rate does not matter.
//
//  * Grid: 32-feature tiles x K-splits.  The K-splits of one tile form a thread-block
//    cluster (<= 8 CTAs): their fp32 partial tiles are summed through distributed shared
//    memory by the cluster's rank-0 CTA in rank order (no global workspace, no atomics,
//    the same sum every run), which then applies the fused epilogue (epilogue.cuh).
//  * Weights: per ring stage, each lane of warp 0 copies one weight-row segment of 128 k
//    with cp.async.bulk (shared rows padded by 16 bytes so ldmatrix is conflict-free),
//    completing on the stage's mbarrier.  Weights never depend on an earlier kernel, so
//    the first stages are issued BEFORE the programmatic-dependent-launch wait and stream
//    in while the preceding kernel of the step finishes.
//  * A operand: after the wait, the CTA's k-range of every row is staged in shared
//    memory, copied (bf16) or standardised from the fp32 residual stream; the row
//    statistics of all rows are reduced in one pass of the block over the full rows.
//  * MMA: mma.sync m16n8k16 bf16 with the weight features as the m16 operand and the
//    tokens as the n8 operand, so a generation step of 8 sequences fills it unpadded.
//  * Every mbarrier wait is bounded (the ring wait by the runtime wait limit, the drain of
//    copies in flight and the cluster reduction by fixed, longer limits); on time-out the CTA
//    records ERRW_TIMEOUT, stops issuing, waits for its copies in flight and still takes part
//    in the cluster barriers, so its cluster always completes.
#define ADEPT_TU_ID 5
#include "gemm_decode.h"
#include "epilogue.cuh"
#include "gemm_tc.h"

#include <cuda.h>

#include <algorithm>
#include <cstring>

namespace adept {
namespace {

constexpr int DG_BN = 32;                        // output features per tile
constexpr int DG_KS = 128;                       // k per ring stage of a short k-range (larger: 256)
constexpr int DG_THREADS = 128;
constexpr int DG_CHUNK = DG_BN * 128;            // bytes of one [32 rows][64 k] 128-byte-swizzled chunk
constexpr int DG_MAX_STAGES = 12;
constexpr int DG_MAX_A = 16 * 2048;              // A-slice elements a CTA holds (rows x k)
constexpr int dg_max_kr(int mb) { return DG_MAX_A / (mb * 8); }   // k per CTA: 4096 (M <= 8), 2048
constexpr int DG_MAX_SPLITS = 8;                 // portable cluster size
constexpr int DG_RP = DG_BN + 1;                 // floats per token row of a partial tile
// Where the fused standardisation takes its row statistics from.
enum : int { DG_STATS_HERE = 0, DG_STATS_ROWS = 1, DG_STATS_TILES = 2 };
constexpr int DG_ROPE_HALF = 64;                 // rotary pairs per row staged for the epilogue (head_dim <= 128)
constexpr int DG_XMAX_BYTES = 64 * 1024;         // fp32 rows staged for the fused standardisation
constexpr long long DG_TIMEOUT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz
// the cluster reduction outlasts any other CTA's bounded waits (its drain included)
constexpr long long DG_REDUCE_TIMEOUT_CYCLES = 16 * DG_TIMEOUT_CYCLES;

// Dynamic shared memory: weight ring | A slice | staged fp32 rows | partial tiles.
struct DgLayout {
  int off_a, off_x, off_t, off_p, total;
};
// Offsets are relative to the ring base (the dynamic shared memory rounded up to 1024
// bytes, as the 128-byte swizzle pattern repeats every 1024 bytes).
constexpr DgLayout dg_layout(int ring, int arows, int kr, int xrows, int xk, int tstats, int splits) {
  return DgLayout{ring, ring + arows * (kr + 8) * 2, ring + arows * (kr + 8) * 2 + xrows * xk * 4,
                  ring + arows * (kr + 8) * 2 + xrows * xk * 4 + xrows * tstats * 8,
                  ring + arows * (kr + 8) * 2 + xrows * xk * 4 + xrows * tstats * 8 + 2 * DG_MAX_M * DG_RP * 4 +
                      (splits - 1) * DG_MAX_M * DG_BN * 4};
}
constexpr int DG_MAX_TSTATS = 128;               // 32-column tiles of a row (d_model <= 4096)
constexpr int DG_STATIC_SMEM = 12 * 1024;          // static shared memory of the kernel (bound)
constexpr int DG_SMEM_LIMIT = 227 * 1024 - DG_STATIC_SMEM;   // dynamic shared memory of one CTA

struct DgParams {
  CUtensorMap wmap;     // W as {64, N, K/64}, box {64, 32, 2}, 128-byte swizzle
  const uint8_t* bt;    // tile-contiguous copy of W (GemmProblem::Bt) or NULL
  int bt_nkb;           // its 256-k blocks per 32-row tile
  const bf16* W;
  int ldw;
  const bf16* A;
  int lda;
  const float* X;       // fused standardisation source (fused_norm)
  int ldx;
  const int* in_rows;
  int norm_mode;
  float eps;
  int fused_norm;
  DevRange rows;
  int N, K;
  int tiles;    // 32-feature tiles
  int splits;   // CTAs per tile (= cluster size)
  int kr;       // k per split (a multiple of ks; the last split may be shorter)
  int ks;       // k per ring stage: 128 or 256 (stage = ks / 64 swizzled chunks)
  int stages;   // ring stages
  int pre;      // stages issued before the grid-dependency wait
  int max_m;    // rows the launch was sized for
  int xrows;    // fp32 rows staged in shared memory for the standardisation (0: streamed)
  int xk;       // staged floats per row: K (statistics computed here) or kr (a k-slice)
  int stat_mode;   // DG_STATS_*
  const float2* row_stats;    // DG_STATS_ROWS: (mu, rstd) per row
  const float2* tile_stats;   // DG_STATS_TILES: [row][n_stiles] (mean, M2) of 32-column tiles
  int n_stiles;
  int off_a, off_x, off_t, off_p;   // dynamic shared-memory offsets (bytes)
  int off_r;                        // rotary epilogues: the rows' (cos, sin) table rows [DG_MAX_M][DG_ROPE_HALF]
  int bias_aligned, resid_aligned;
  Epi epi;
  unsigned* err;
  SpanCtx span;
};

// Several problems of one launch that differ only in the weights, the row range and the
// epilogue (the grouped skipped-layer fill: one problem per layer), blockIdx.y = problem.
constexpr int DG_MAX_GROUPS = 32;
struct DgParamsG : DgParams {
  CUtensorMap gmap[DG_MAX_GROUPS];
  const uint8_t* gbt[DG_MAX_GROUPS];
  DevRange grows[DG_MAX_GROUPS];
  Epi gepi[DG_MAX_GROUPS];
};
__device__ __forceinline__ const CUtensorMap* dg_wmap(const DgParams& p) { return &p.wmap; }
__device__ __forceinline__ const uint8_t* dg_bt(const DgParams& p) { return p.bt; }
__device__ __forceinline__ const uint8_t* dg_bt(const DgParamsG& p) { return p.gbt[blockIdx.y]; }
__device__ __forceinline__ const CUtensorMap* dg_wmap(const DgParamsG& p) { return &p.gmap[blockIdx.y]; }
__device__ __forceinline__ DevRange dg_rows(const DgParams& p) { return p.rows; }
__device__ __forceinline__ DevRange dg_rows(const DgParamsG& p) { return p.grows[blockIdx.y]; }
__device__ __forceinline__ const Epi& dg_epi(const DgParams& p) { return p.epi; }
__device__ __forceinline__ const Epi& dg_epi(const DgParamsG& p) { return p.gepi[blockIdx.y]; }

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
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
__device__ __forceinline__ bool dg_wait(uint64_t* bar, uint32_t parity, unsigned* err, long long limit) {
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
// Wait with acquire at cluster scope (arrivals from other CTAs of the cluster).
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool dg_wait_cluster(uint64_t* bar, uint32_t parity, unsigned* err, long long limit) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait_cluster(bar, parity)) {
    if (clock64() - t0 > limit) {
      atomicOr(err, ERRW_TIMEOUT);
      return false;
    }
  }
  return true;
}
// 16-byte store into the shared memory of cluster CTA `rank` (at this CTA's offset of dst),
// completing its bytes on that CTA's mbarrier at this CTA's offset of bar.
__device__ __forceinline__ void st_async_v4(float* dst, const float4& v, uint64_t* bar, uint32_t rank) {
  uint32_t rd, rb;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rd) : "r"(smem_u32(dst)), "r"(rank));
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rb) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(rd),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rb)
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
__device__ __forceinline__ void tma_load_3d(const CUtensorMap* tm, uint64_t* bar, void* dst, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::
          "r"(smem_u32(dst)),
      "l"((uint64_t)tm), "r"(0), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
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
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// MB: 8-token blocks of the A operand (1: M <= 8, 2: M <= 16); KIND: the epilogue kind.
template <int MB, int KIND, class P = DgParams>
__global__ void __launch_bounds__(DG_THREADS, 1) gemm_decode_kernel(const __grid_constant__ P p) {
  KT_BEGIN();
  extern __shared__ __align__(128) uint8_t dg_smem_raw[];
  __shared__ __align__(8) uint64_t full[DG_MAX_STAGES];
  __shared__ __align__(8) uint64_t red_bar;          // leader: one arrival per other split
  __shared__ __align__(16) float s_bias[DG_BN];
  __shared__ __align__(16) float s_res[DG_MAX_M][DG_BN];
  __shared__ EpiRow s_rr[DG_MAX_M];
  __shared__ float s_red[DG_THREADS / 32][MB * 8];
  __shared__ float s_mu[MB * 8], s_rs[MB * 8];
  __shared__ unsigned s_span_left;
  __shared__ unsigned long long s_span_t0;
  SpanScope span(p.span, &s_span_left, &s_span_t0);

  const long long wlim = wait_limit();   // the runtime wait limit, read once
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // tiles tile0, tile0 + tstride, ... of one K-split (several only when splits == 1)
  const int tile0 = blockIdx.x / p.splits, split = blockIdx.x - tile0 * p.splits;
  const int tstride = gridDim.x / p.splits;
  const int my_tiles = (p.tiles - tile0 + tstride - 1) / tstride;
  const int k_lo = split * p.kr;
  const int kr = min(p.K - k_lo, p.kr);
  const int ks = p.ks, stage_bytes = ks * DG_BN * 2;
  const int nst = (kr + ks - 1) / ks;   // stages per tile
  const int G = my_tiles * nst;               // stages of this CTA
  const int S = p.stages;
  const int apitch = p.kr + 8;           // A row pitch in elements (16-byte shift per row)
  uint8_t* dg_smem = dg_smem_raw + ((1024 - (smem_u32(dg_smem_raw) & 1023)) & 1023);
  uint8_t* sW = dg_smem;                                                // [S][2][32 rows][128 B], swizzled
  bf16* sA = reinterpret_cast<bf16*>(dg_smem + p.off_a);                // [16 (MB 2) or max_m rows][apitch]
  float* sX = reinterpret_cast<float*>(dg_smem + p.off_x);              // [xrows][xk] (fused standardisation)
  float2* sT = reinterpret_cast<float2*>(dg_smem + p.off_t);            // [xrows][n_stiles] producer tile stats
  constexpr int SLOT = DG_MAX_M * DG_RP;
  float* sP = reinterpret_cast<float*>(dg_smem + p.off_p);              // [2][DG_MAX_M][DG_RP]: own k halves
  float* sR = sP + 2 * SLOT;                                            // [splits - 1][DG_MAX_M][32]: pushed
  // rotary epilogues only (kept out of the other kernels' footprint, so that more of their
  // CTAs fit beside a neighbouring launch's)
  float2 (*s_rope)[DG_ROPE_HALF] = reinterpret_cast<float2 (*)[DG_ROPE_HALF]>(dg_smem + p.off_r);
  const uint32_t rank = p.splits > 1 ? cluster_rank() : 0u;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&full[s], 1);
    mbar_init(&red_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // the leader's reduction barrier completes when every other split has pushed its
    // partial tile (MB*8 rows x 32 features, whatever the row count)
    if (p.splits > 1 && rank == 0) mbar_expect_tx(&red_bar, (uint32_t)((p.splits - 1) * MB * 8 * DG_BN * 4));
  }
  span.init();
  __syncthreads();
  pdl_launch_dependents();

  // warp 0 lane 0: stage g of this CTA (tile g / nst, k-block g % nst) into ring slot g % S,
  // one TMA copy of 32 rows x 128 k (rows past N and k past K arrive as zeros)
  auto issue = [&](int g) {
    if (lane != 0) return;
    const int j = g / nst, kb = g - j * nst;
    const int f = (tile0 + j * tstride) * DG_BN;
    const int s = g % S;
    mbar_expect_tx(&full[s], (uint32_t)stage_bytes);
    const uint8_t* bt = dg_bt(p);
    if (bt) {   // the stage's chunks are contiguous within one 16 KB unit of the tiled copy
      const int k = k_lo + kb * ks;
      bulk_load(sW + (size_t)s * stage_bytes,
                bt + ((size_t)(f >> 5) * p.bt_nkb + (k >> 8)) * (32 * 256 * 2) + ((k & 255) >> 6) * DG_CHUNK,
                (uint32_t)stage_bytes, &full[s]);
    } else {
      tma_load_3d(dg_wmap(p), &full[s], sW + (size_t)s * stage_bytes, f, (k_lo + kb * ks) >> 6);
    }
  };
  const int first = min(S, G);
  const int pre = min(p.pre, first);
  if (warp == 0)
    for (int g = 0; g < pre; ++g) issue(g);
  // every CTA's reduction barrier is initialised before another CTA of the cluster can arrive on it
  if (p.splits > 1) cluster_sync();

  pdl_wait();   // from here on, the preceding kernels' writes are visible
  KT_WAITED();
  span.waited();

  const DevRange prow = dg_rows(p);
  const int rb = prow.b();
  int M = prow.e() - rb;
  if (M > p.max_m) {   // more rows than the launch was sized for
    if (tid == 0) atomicOr(p.err, ERRW_CONFIG);
    M = p.max_m;
  }
  if (M <= 0) {
    // no rows (every token of the step has left): let the copies in flight land, leave
    // (M is the same in every CTA of the cluster, so no CTA waits for another)
    if (warp == 0)
      for (int g = 0; g < pre; ++g) dg_wait(&full[g], 0, p.err, DG_TIMEOUT_CYCLES);
    return;
  }
  if (warp == 0)
    for (int g = pre; g < first; ++g) issue(g);
  KT_MARK(0);

  // ---- one round trip: operand rows (warps 0-2) and the epilogue's inputs (warp 3)
  const Epi& e = dg_epi(p);
  const bool leader = rank == 0;
  // bias and residual columns are staged for a CTA with a single full tile
  const bool single = my_tiles == 1 && (tile0 + 1) * DG_BN <= p.N;
  const int f_single = tile0 * DG_BN;
  const bool st_bias = leader && single && e.bias && p.bias_aligned;
  const bool st_res = leader && single && e.kind == EPI_RESID && p.resid_aligned;
  const bool st_rows = leader && (e.kind == EPI_QKV || e.kind == EPI_KV);
  if (warp < 3) {
    const int t = tid;   // 0..95
    if (p.fused_norm && p.xrows) {
      // fp32 rows: whole (statistics computed here) or only the k-slice (statistics from
      // the producer), and the producer's per-tile statistics
      int src[MB * 8];
#pragma unroll
      for (int r = 0; r < MB * 8; ++r) src[r] = r < M ? (p.in_rows ? p.in_rows[rb + r] : rb + r) : 0;
      const int x0 = p.stat_mode == DG_STATS_HERE ? 0 : k_lo;
      const int cpr = (p.stat_mode == DG_STATS_HERE ? p.K : kr) >> 2;   // 16-byte chunks per row
#pragma unroll
      for (int r = 0; r < MB * 8; ++r) {
        if (r >= M) break;
        const float* x = p.X + (size_t)src[r] * p.ldx + x0;
        for (int c = t; c < cpr; c += 96) cp_async16(sX + (size_t)r * p.xk + c * 4, x + c * 4);
      }
      if (p.stat_mode == DG_STATS_TILES)
        for (int c = t; c < M * (p.n_stiles >> 1); c += 96) {
          const int r = c / (p.n_stiles >> 1), q = c - r * (p.n_stiles >> 1);
          cp_async16(sT + (size_t)r * p.n_stiles + q * 2, p.tile_stats + (size_t)(rb + r) * p.n_stiles + q * 2);
        }
    } else if (!p.fused_norm) {
      const int cpr = kr >> 3;   // 16-byte chunks per bf16 row
      for (int r = 0; r < M; ++r) {
        const bf16* a = p.A + (size_t)(rb + r) * p.lda + k_lo;
        for (int c = t; c < cpr; c += 96) cp_async16(sA + r * apitch + c * 8, a + c * 8);
      }
    }
  } else {
    if (p.fused_norm && p.stat_mode == DG_STATS_ROWS && lane < M) {
      const float2 st = p.row_stats[rb + lane];
      s_mu[lane] = st.x;
      s_rs[lane] = st.y;
    }
    if (st_bias && lane < DG_BN / 4) cp_async16(s_bias + lane * 4, e.bias + f_single + lane * 4);
    if (st_res)
      for (int c = lane; c < M * (DG_BN / 4); c += 32) {
        const int r = c >> 3, q = c & 7;
        cp_async16(&s_res[r][q * 4], e.resid + (size_t)(rb + r) * e.ld_resid + f_single + q * 4);
      }
    if (st_rows && lane < M) {
      EpiRow rr = epi_row(e, rb + lane);
      if (e.rope) {   // the row's whole (cos, sin) table row: every tile of the CTA reads it
        const int half = e.head_dim >> 1;
        const float2* tab = e.rope_table + (size_t)rr.pos * half;
        for (int c = 0; c < half / 2; ++c) cp_async16(&s_rope[lane][c * 2], tab + c * 2);
        rr.rope = s_rope[lane];
      }
      s_rr[lane] = rr;
    }
  }
  cp_async_wait_all();
  __syncthreads();
  KT_MARK(1);

  // ---- fused standardisation of the A operand (gains live in W)
  if (p.fused_norm) {
    const int K = p.K;
    if (p.xrows) {
      // rows padded to 2^lg; tpr = 128 >> lg threads per row, float4 reads
      const int lg = M > 8 ? 4 : M > 4 ? 3 : M > 2 ? 2 : M > 1 ? 1 : 0;
      const int tpr = DG_THREADS >> lg;
      const int r = tid >> (7 - lg), sub = tid & (tpr - 1);
      const bool live = r < M;
      const float4* x4 = reinterpret_cast<const float4*>(sX + (size_t)(live ? r : 0) * p.xk);
      if (p.stat_mode == DG_STATS_HERE) {
        const int K4 = K >> 2;
        // sum over the row's tpr threads (shuffles within a warp, shared memory across warps)
        auto group_sum = [&](float v) {
          if (tpr <= 32) {
            for (int o = tpr >> 1; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            return v;
          }
          v = warp_sum(v);
          if (lane == 0) s_red[warp][0] = v;
          __syncthreads();
          const int w0 = (tid / tpr) * (tpr >> 5);
          float t = 0.f;
          for (int w = 0; w < (tpr >> 5); ++w) t += s_red[w0 + w][0];
          __syncthreads();
          return t;
        };
        float mu = 0.f, rs = 1.f;
        if (p.norm_mode == NORM_LN) {
          float a0 = 0.f, a1 = 0.f;
          if (live)
            for (int v = sub; v < K4; v += tpr) {
              const float4 t = x4[v];
              a0 += t.x + t.y;
              a1 += t.z + t.w;
            }
          mu = group_sum(a0 + a1) / K;
        }
        if (p.norm_mode != NORM_COPY) {
          float a0 = 0.f, a1 = 0.f;
          if (live)
            for (int v = sub; v < K4; v += tpr) {
              const float4 t = x4[v];
              const float c0 = t.x - mu, c1 = t.y - mu, c2 = t.z - mu, c3 = t.w - mu;
              a0 += c0 * c0 + c1 * c1;
              a1 += c2 * c2 + c3 * c3;
            }
          rs = rsqrtf(group_sum(a0 + a1) / K + p.eps);
        }
        if (live && sub == 0) {
          s_mu[r] = mu;
          s_rs[r] = rs;
        }
      } else if (p.stat_mode == DG_STATS_TILES) {
        // the row's moments from the producer's 32-column (mean, M2) tiles, about the first
        // tile's mean c: S1 = sum 32 (m_t - c), S2 = sum M2_t + 32 (m_t - c)^2; warp w takes
        // rows w, w + 4, ..., lane l tiles l, l + 32, ...
        for (int r2 = warp; r2 < M; r2 += 4) {
          const float2* ts = sT + (size_t)r2 * p.n_stiles;
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
            s_mu[r2] = mu;
            s_rs[r2] = rs;
          }
        }
      }
      __syncthreads();
      if (live) {
        const float mu = s_mu[r], rs = s_rs[r];
        const int xoff = p.stat_mode == DG_STATS_HERE ? (k_lo >> 2) : 0;
        for (int v = sub; v < (kr >> 2); v += tpr) {
          const float4 t = x4[xoff + v];
          const __nv_bfloat162 lo = __floats2bfloat162_rn((t.x - mu) * rs, (t.y - mu) * rs);
          const __nv_bfloat162 hi = __floats2bfloat162_rn((t.z - mu) * rs, (t.w - mu) * rs);
          uint2 u;
          u.x = *reinterpret_cast<const uint32_t*>(&lo);
          u.y = *reinterpret_cast<const uint32_t*>(&hi);
          *reinterpret_cast<uint2*>(sA + r * apitch + v * 4) = u;
        }
      }
    } else {
      // rows too long to stage: block sums over global memory, all rows at once
      const float* xr[MB * 8];
#pragma unroll
      for (int r = 0; r < MB * 8; ++r) {
        const int src = r < M ? (p.in_rows ? p.in_rows[rb + r] : rb + r) : 0;
        xr[r] = p.X + (size_t)src * p.ldx;
      }
      auto row_sums = [&](auto term, float* out) {
        float part[MB * 8];
#pragma unroll
        for (int r = 0; r < MB * 8; ++r) part[r] = 0.f;
        for (int d = tid; d < K; d += DG_THREADS) {
#pragma unroll
          for (int r = 0; r < MB * 8; ++r)
            if (r < M) part[r] += term(r, xr[r][d]);
        }
#pragma unroll
        for (int r = 0; r < MB * 8; ++r) {
          const float v = warp_sum(part[r]);
          if (lane == 0) s_red[warp][r] = v;
        }
        __syncthreads();
        if (tid < MB * 8) out[tid] = (s_red[0][tid] + s_red[1][tid] + s_red[2][tid] + s_red[3][tid]) / K;
        __syncthreads();
      };
      if (tid < MB * 8) {
        s_mu[tid] = 0.f;
        s_rs[tid] = 1.f;
      }
      __syncthreads();
      if (p.norm_mode == NORM_LN) row_sums([](int, float x) { return x; }, s_mu);
      if (p.norm_mode != NORM_COPY) {
        row_sums([&](int r, float x) { const float c = x - s_mu[r]; return c * c; }, s_rs);
        if (tid < MB * 8) s_rs[tid] = rsqrtf(s_rs[tid] + p.eps);
        __syncthreads();
      }
#pragma unroll
      for (int r = 0; r < MB * 8; ++r) {
        if (r >= M) break;
        const float mu = s_mu[r], rs = s_rs[r];
        const float* x = xr[r] + k_lo;
        for (int k = 2 * tid; k < kr; k += 2 * DG_THREADS)
          *reinterpret_cast<__nv_bfloat162*>(sA + r * apitch + k) =
              __floats2bfloat162_rn((x[k] - mu) * rs, (x[k + 1] - mu) * rs);
      }
    }
    __syncthreads();
  }

  KT_MARK(2);

  // ---- tiles: main loop, partial tile, (cluster) reduction, epilogue
  const int mb = warp & 1, kh = warp >> 1;
  // weight fragment rows of this lane; k-chunk kh of the stage; 16-byte unit u of a
  // 128-byte row sits at (u ^ (row & 7)) * 16
  const int wrow = mb * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
  const uint32_t w_base = smem_u32(sW) + kh * DG_CHUNK + wrow * 128;
  const int wx = wrow & 7, wu = (lane >> 4) & 1;
  const uint32_t a_base = smem_u32(sA) + ((lane & 7) + ((lane >> 4) & 1) * 8) * apitch * 2 + ((lane >> 3) & 1) * 16 +
                          kh * 128;
  // MB == 1: lane (g, t) of the m16n8k16 B fragment reads row g, k 2t (+8) of each k16 step
  const int bg = lane >> 2;
  const uint32_t b_base = smem_u32(sA) + (bg * apitch + kh * 64 + (lane & 3) * 2) * 2;
  int dead = 0, g = 0;
  for (int j = 0; j < my_tiles && !dead; ++j) {
    const int f0 = (tile0 + j * tstride) * DG_BN;
    float acc[MB][4];
#pragma unroll
    for (int t = 0; t < MB; ++t) acc[t][0] = acc[t][1] = acc[t][2] = acc[t][3] = 0.f;
    for (int kb = 0; kb < nst; ++kb, ++g) {
      const int s = g % S;
#ifdef ADEPT_KTRACE
      const unsigned long long tw = kt_now();
#endif
      // every lane polls (it leaves the wait as soon as the stage lands); one vote makes the
      // outcome warp-uniform, since the MMAs below are .aligned
      const bool ok = __all_sync(0xffffffffu, dg_wait(&full[s], (uint32_t)((g / S) & 1), p.err, wlim)) != 0;
#ifdef ADEPT_KTRACE
      KT_ADD(7, kt_now() - tw);
#endif
      // warp (mb, kh) takes the stage's 64-k chunks kh, kh + 2, ...
      const int nch = min(ks, kr - kb * ks) >> 6;
      for (int q = 0; ok && 2 * q + kh < nch; ++q) {
        const uint32_t wa = w_base + s * stage_bytes + q * (2 * DG_CHUNK);
        const uint32_t aa = a_base + (kb * ks + q * 128) * 2;
        const uint32_t ab = b_base + (kb * ks + q * 128) * 2;
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
            // n8 block of at most 8 rows: fragment words loaded directly, rows >= M zero
            // (the A slice holds only the launch's rows)
            uint32_t b0 = 0u, b1 = 0u;
            if (bg < M) {
              b0 = ld_shared_u32(ab + kk * 32);
              b1 = ld_shared_u32(ab + kk * 32 + 16);
            }
            mma_bf16(acc[0], a, b0, b1);
          }
        }
      }
      if (__syncthreads_or(!ok)) {   // every warp is done with slot s
        dead = 1;
        break;
      }
      if (warp == 0 && g + S < G) issue(g + S);
    }
    if (dead) {
      if (warp == 0)   // stop: wait (bounded) for the copies still in flight
        for (int h = g; h < min(G, g + S); ++h) dg_wait(&full[h % S], (uint32_t)((h / S) & 1), p.err, DG_TIMEOUT_CYCLES);
      if (p.splits == 1) return;
    }
    KT_MARK(3);

    // partial tile [token][feature] of this CTA (sum of the two k halves) in slot 0
    {
      float* part = sP + kh * SLOT;
      const int gq = lane >> 2, t4 = lane & 3;
#pragma unroll
      for (int t = 0; t < MB; ++t) {
        const int tk = t * 8 + 2 * t4, fc = mb * 16 + gq;
        part[tk * DG_RP + fc] = acc[t][0];
        part[(tk + 1) * DG_RP + fc] = acc[t][1];
        part[tk * DG_RP + fc + 8] = acc[t][2];
        part[(tk + 1) * DG_RP + fc + 8] = acc[t][3];
      }
    }
    __syncthreads();
    if (p.splits > 1 && !leader) {
      // push the partial tile (dense rows of 32) into slot rank - 1 of the leader; the
      // bytes complete on the leader's reduction barrier
      for (int q = tid; q < MB * 8 * (DG_BN / 4); q += DG_THREADS) {
        const int row = q >> 3, c = (q & 7) * 4, i = row * DG_RP + c;
        const float4 v = make_float4(sP[i] + sP[SLOT + i], sP[i + 1] + sP[SLOT + i + 1], sP[i + 2] + sP[SLOT + i + 2],
                                     sP[i + 3] + sP[SLOT + i + 3]);
        st_async_v4(sR + (rank - 1) * (DG_MAX_M * DG_BN) + row * DG_BN + c, v, &red_bar, 0u);
      }
      return;
    }
    for (int e2 = tid; e2 < M * DG_BN; e2 += DG_THREADS) {
      const int i = (e2 >> 5) * DG_RP + (e2 & 31);
      sP[i] += sP[SLOT + i];
    }
    if (p.splits > 1) {
      // leader: the other splits' partials, summed in rank order
      const bool ok = dg_wait_cluster(&red_bar, 0u, p.err, DG_REDUCE_TIMEOUT_CYCLES);
      if (__syncthreads_or(!ok)) dead = 1;
      for (int e2 = tid; e2 < M * DG_BN; e2 += DG_THREADS) {
        const int i = (e2 >> 5) * DG_RP + (e2 & 31);
        float v = sP[i];
        for (int r = 1; r < p.splits; ++r) v += sR[(r - 1) * (DG_MAX_M * DG_BN) + e2];
        sP[i] = v;
      }
    }
    __syncthreads();
    KT_MARK(4);
    if (dead) return;

    // fused epilogue, element-parallel: warp w takes rows w, w + 4, ..., lane = feature
    KT_MARK(5);
    for (int row = warp; row < M; row += 4) {
      const int ra = rb + row, c = f0 + lane;
      const bool valid = c < p.N;
      float v = sP[row * DG_RP + lane];
      if (e.bias && valid) v += st_bias ? s_bias[lane] : e.bias[c];
      if (KIND == EPI_F32) {
        if (valid) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
      } else if (KIND == EPI_ACT) {
        v = apply_act(e.act, v);
        if (valid) {
          ((bf16*)e.out_t)[(size_t)ra * e.ld_t + c] = __float2bfloat16_rn(v);
          if (e.out_f32) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
        }
      } else if (KIND == EPI_RESID) {
        if (valid) v += st_res ? s_res[row][lane] : e.resid[(size_t)ra * e.ld_resid + c];
        if (valid) e.out_f32[(size_t)ra * e.ld_f32 + c] = v;
        if (e.tile_stats) {   // (mean, M2) of the row's 32 results (full tiles: N % 32 == 0)
          const float mean = warp_sum(v) * (1.f / DG_BN);
          const float m2 = warp_sum((v - mean) * (v - mean));
          if (lane == 0) e.tile_stats[(size_t)ra * (p.N / DG_BN) + f0 / DG_BN] = make_float2(mean, m2);
        }
      } else if (KIND == EPI_SWIGLU) {
        // features interleaved in blocks of 16: lanes 0-15 gate, 16-31 the matching up
        const float u = __shfl_down_sync(0xffffffffu, v, 16);
        if (lane < 16) ((bf16*)e.out_t)[(size_t)ra * e.ld_t + (f0 >> 1) + lane] = __float2bfloat16_rn(silu_f(v) * u);
      } else {   // EPI_QKV / EPI_KV: q -> out_t, k / v -> the row's cache slot; RoPE pairs adjacent
        const EpiRow rr = st_rows ? s_rr[row] : epi_row(e, ra);
        const int dh = e.head_dim, half = dh >> 1, nq = e.n_q_cols, nkv = e.n_kv_cols;
        const int base = c < nq ? 0 : c < nq + nkv ? nq : nq + nkv;
        const int hd = (c - base) / dh, d = (c - base) - hd * dh;
        const float pv = __shfl_xor_sync(0xffffffffu, v, 1);   // the other member of the pair
        float o = v;
        int od = d;
        if (e.rope && base < nq + nkv) {
          const int ip = d >> 1;
          const float2 cs = rr.rope ? rr.rope[ip] : e.rope_table[(size_t)rr.pos * half + ip];
          // (x1, x2) = (even, odd) column of the pair -> x1 c - x2 s at ip, x2 c + x1 s at ip + half
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
    KT_MARK(6);
    __syncthreads();   // slot 0 is rewritten by the next tile
  }
}


int g_dg_sms = 0;

template <int MB, int KIND>
cudaError_t launch_dg(cudaStream_t st, const DgParams& prm, int grid, size_t smem) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(gemm_decode_kernel<MB, KIND>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, DG_SMEM_LIMIT);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(DG_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (prm.splits > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = prm.splits;
    at[na].val.clusterDim.y = 1;
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
  return cudaLaunchKernelEx(&cfg, gemm_decode_kernel<MB, KIND>, prm);
}

// Grouped launch (EPI_KV problems): grid (gx, groups), clusters along x.
template <int MB>
cudaError_t launch_dg_grouped(cudaStream_t st, const DgParamsG& prm, int gx, int groups, size_t smem) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(gemm_decode_kernel<MB, EPI_KV, DgParamsG>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, DG_SMEM_LIMIT);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(gx, groups);
  cfg.blockDim = dim3(DG_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (prm.splits > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = prm.splits;
    at[na].val.clusterDim.y = 1;
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
  return cudaLaunchKernelEx(&cfg, gemm_decode_kernel<MB, EPI_KV, DgParamsG>, prm);
}

template <int MB>
cudaError_t launch_kind(cudaStream_t st, const DgParams& prm, int grid, size_t smem) {
  switch (prm.epi.kind) {
    case EPI_F32: return launch_dg<MB, EPI_F32>(st, prm, grid, smem);
    case EPI_ACT: return launch_dg<MB, EPI_ACT>(st, prm, grid, smem);
    case EPI_RESID: return launch_dg<MB, EPI_RESID>(st, prm, grid, smem);
    case EPI_SWIGLU: return launch_dg<MB, EPI_SWIGLU>(st, prm, grid, smem);
    case EPI_QKV: return launch_dg<MB, EPI_QKV>(st, prm, grid, smem);
    default: return launch_dg<MB, EPI_KV>(st, prm, grid, smem);
  }
}

}  // namespace

bool decode_gemm_supported(const GemmProblem& q, int max_rows, const DgNorm* norm) {
  if (max_rows <= 0 || max_rows > DG_MAX_M) return false;
  if (q.N <= 0 || q.K <= 0 || q.K % 64 || q.K > DG_MAX_SPLITS * dg_max_kr(max_rows > 8 ? 2 : 1)) return false;
  if (q.ldb % 8 || ((uintptr_t)q.B & 15)) return false;
  if (!norm && (q.lda % 8 || ((uintptr_t)q.A & 15))) return false;
  if (norm && !norm->X) return false;
  if ((q.epi.kind == EPI_QKV || q.epi.kind == EPI_KV || q.epi.kind == EPI_SWIGLU) && q.N % 32) return false;
  if (q.epi.rope && (q.epi.head_dim > 2 * DG_ROPE_HALF || q.epi.head_dim % 4)) return false;
  if (q.epi.kind < EPI_F32 || q.epi.kind > EPI_KV) return false;
  if (q.epi.tile_stats && (q.epi.kind != EPI_RESID || q.N % DG_BN)) return false;
  if (norm && norm->tile_stats && (q.K % 64 || ((uintptr_t)norm->tile_stats & 15))) return false;
  return true;
}

// Launch plan of one problem (or of `groups` problems of the same shape, one per gridDim.y):
// fills prm (except the tensor map) and the x-grid, dynamic shared memory and row blocks.
static bool dg_plan(const GemmProblem& q, int max_rows, const DgNorm* norm, int groups, unsigned* err, DgParams& prm,
                    int& grid_out, size_t& smem_out, int& mb_out) {
  if (!decode_gemm_supported(q, max_rows, norm)) return false;
  if (!g_dg_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_dg_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_dg_sms <= 0) g_dg_sms = 1;
  }
  const int tiles = cdiv(q.N, DG_BN);
  const int mb = max_rows > 8 ? 2 : 1;
  const int kr_max = dg_max_kr(mb);
  // K-splits: enough CTAs to cover the GPU about twice, each split at least one stage and
  // at most kr_max of k
  int splits = std::max(cdiv(2 * g_dg_sms, tiles * groups), cdiv(q.K, kr_max));
  splits = std::min(splits, std::min(DG_MAX_SPLITS, cdiv(q.K, DG_KS)));
  // long k-ranges split over a cluster stage 256 k per row (512 contiguous bytes of each
  // weight row per copy); a single split keeps 128 k, which leaves room for more resident
  // CTAs of the persistent grid (measured faster at the Llama-7B QKV shape)
  const int ks = splits > 1 && cdiv(q.K, splits) >= 1024 ? 2 * DG_KS : DG_KS;
  const int kr = cdiv(cdiv(q.K, splits), ks) * ks;
  if (kr > kr_max) return false;
  splits = cdiv(q.K, kr);
  const int nst = kr / ks;
  const int stage_bytes = ks * DG_BN * 2;
  prm.W = (const bf16*)q.B;
  prm.ldw = q.ldb;
  prm.A = (const bf16*)q.A;
  prm.lda = q.lda;
  prm.X = norm ? norm->X : nullptr;
  prm.ldx = norm ? norm->ldx : 0;
  prm.in_rows = norm ? norm->in_rows : nullptr;
  prm.norm_mode = norm ? norm->mode : NORM_COPY;
  prm.eps = norm ? norm->eps : 0.f;
  prm.fused_norm = norm != nullptr;
  prm.rows = q.rows;
  prm.N = q.N;
  prm.K = q.K;
  prm.tiles = tiles;
  prm.splits = splits;
  prm.kr = kr;
  prm.ks = ks;
  prm.max_m = max_rows;
  // statistics from the producer when given (only the k-slice of each row is staged),
  // else computed here from whole staged rows (or, rows too long to stage, streamed)
  prm.stat_mode = !norm                                             ? DG_STATS_HERE
                  : norm->row_stats                                 ? DG_STATS_ROWS
                  : norm->tile_stats && q.K / 32 <= DG_MAX_TSTATS ? DG_STATS_TILES
                                                                    : DG_STATS_HERE;
  prm.row_stats = norm ? norm->row_stats : nullptr;
  prm.tile_stats = norm ? norm->tile_stats : nullptr;
  prm.n_stiles = q.K / 32;
  prm.xk = prm.stat_mode == DG_STATS_HERE ? q.K : kr;
  const bool x_ok = norm && norm->ldx % 4 == 0 && ((uintptr_t)norm->X & 15) == 0;
  prm.xrows = x_ok && (size_t)max_rows * prm.xk * 4 <= (size_t)DG_XMAX_BYTES ? max_rows : 0;
  if (prm.xrows == 0) prm.stat_mode = DG_STATS_HERE;   // the streamed path computes its own
  // grid: one K-split -> persistent CTAs streaming their tiles' weights through their
  // rings; several splits -> one CTA per (tile, split)
  const int arows = mb == 2 ? 16 : max_rows;   // A-slice rows held in shared memory
  const int tst = prm.stat_mode == DG_STATS_TILES ? prm.n_stiles : 0;
  const int rope_bytes = q.epi.rope ? DG_MAX_M * DG_ROPE_HALF * (int)sizeof(float2) : 0;
  const int fixed0 = ((dg_layout(0, arows, kr, prm.xrows, prm.xk, tst, splits).total + 15) & ~15) + rope_bytes + 1024;
  int grid = tiles * splits;
  if (splits == 1 && groups == 1) {
    // as many CTAs as can be resident with a ring of at least four stages, each with the
    // same number of tiles (so that no CTA streams a tile while the others idle)
    const int cap = std::max(1, std::min(4, (227 * 1024) / (fixed0 + 4 * stage_bytes + DG_STATIC_SMEM))) * g_dg_sms;
    const int per_cta = cdiv(tiles, cap);
    grid = cdiv(tiles, per_cta);
  }
  const int per_sm = std::min(4, cdiv(grid * groups, g_dg_sms));
  // ring stages: as many as the CTAs resident on an SM leave room for (at most the CTA's
  // stage count), so that the weight bytes in flight cover the memory latency
  const int cta_stages = cdiv(tiles, grid / splits) * nst;
  int stages = (227 * 1024 / per_sm - DG_STATIC_SMEM - fixed0) / stage_bytes;
  stages = std::max(1, std::min(stages, std::min(DG_MAX_STAGES, cta_stages)));
  const DgLayout L = dg_layout(stages * stage_bytes, arows, kr, prm.xrows, prm.xk, tst, splits);
  const int off_r = (L.total + 15) & ~15;
  const size_t smem = (size_t)off_r + rope_bytes + 1024;   // + slack to align the ring to 1024 bytes
  if (smem > (size_t)DG_SMEM_LIMIT) return false;
  prm.stages = stages;
  prm.off_a = L.off_a;
  prm.off_x = L.off_x;
  prm.off_t = L.off_t;
  prm.off_p = L.off_p;
  prm.off_r = off_r;
  prm.bias_aligned = ((uintptr_t)q.epi.bias & 15) == 0;
  prm.resid_aligned = ((uintptr_t)q.epi.resid & 15) == 0 && q.epi.ld_resid % 4 == 0;
  prm.epi = q.epi;
  prm.err = err;
  prm.span = g_span;
  // a CTA whose stages fit the ring issues them all before the grid-dependency wait; a
  // longer one (large models) only its first, which bounds the weight traffic of a layer
  // whose rows have all left
  prm.pre = cta_stages <= stages ? stages : 1;
  grid_out = grid;
  smem_out = smem;
  mb_out = mb;
  return true;
}

// The problem's tile-contiguous copy when every stage of the plan lies inside one unit of it (a
// k-range starting on a multiple of the stage width, which divides 256), else NULL.
static const uint8_t* dg_tiled(const GemmProblem& q, const DgParams& prm) {
  if (!q.Bt || q.bt_nkb != cdiv(q.K, 256) || ((uintptr_t)q.Bt & 15)) return nullptr;
  if (256 % prm.ks || prm.kr % prm.ks) return nullptr;
  return (const uint8_t*)q.Bt;
}

int decode_gemm(cudaStream_t st, const GemmProblem& q, int max_rows, const DgNorm* norm, unsigned* err) {
  thread_local DgParams prm;   // 64-byte-aligned tensor map; one per host thread
  memset(&prm, 0, sizeof prm);
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!dg_plan(q, max_rows, norm, 1, err, prm, grid, smem, mb)) return -1;
  if (!tc_encode_weight_3d(&prm.wmap, q.B, q.K, q.N, (size_t)q.ldb * 2, DG_BN, prm.ks / 64)) return -1;
  prm.bt = dg_tiled(q, prm);
  prm.bt_nkb = q.bt_nkb;
  const cudaError_t e = mb == 2 ? launch_kind<2>(st, prm, grid, smem) : launch_kind<1>(st, prm, grid, smem);
  return e == cudaSuccess ? 1 : -1;
}

int decode_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n, int max_rows, unsigned* err) {
  if (n < 1 || n > DG_MAX_GROUPS) return -1;
  const GemmProblem& q0 = probs[0];
  for (int i = 0; i < n; ++i) {
    const GemmProblem& q = probs[i];
    if (q.epi.kind != EPI_KV || q.A != q0.A || q.lda != q0.lda || q.N != q0.N || q.K != q0.K || q.ldb != q0.ldb ||
        q.epi.rope != q0.epi.rope || q.rows.begin != nullptr || !decode_gemm_supported(q, max_rows, nullptr))
      return -1;
  }
  thread_local DgParamsG prm;   // one per host thread
  memset(&prm, 0, sizeof prm);
  int grid = 0, mb = 1;
  size_t smem = 0;
  if (!dg_plan(q0, max_rows, nullptr, n, err, prm, grid, smem, mb)) return -1;
  for (int i = 0; i < n; ++i) {
    if (!tc_encode_weight_3d(&prm.gmap[i], probs[i].B, q0.K, q0.N, (size_t)q0.ldb * 2, DG_BN, prm.ks / 64)) return -1;
    prm.grows[i] = probs[i].rows;
    prm.gepi[i] = probs[i].epi;
    prm.gepi[i].tile_stats = nullptr;
  }
  // the tiled copies, if every problem of the launch has one (all problems read the same way)
  bool all_tiled = true;
  for (int i = 0; i < n; ++i) all_tiled &= dg_tiled(probs[i], prm) != nullptr;
  for (int i = 0; i < n; ++i) prm.gbt[i] = all_tiled ? dg_tiled(probs[i], prm) : nullptr;
  prm.bt_nkb = q0.bt_nkb;
  prm.bias_aligned = 1;
  for (int i = 0; i < n; ++i) prm.bias_aligned &= ((uintptr_t)probs[i].epi.bias & 15) == 0;
  const cudaError_t e = mb == 2 ? launch_dg_grouped<2>(st, prm, grid, n, smem) : launch_dg_grouped<1>(st, prm, grid, n, smem);
  return e == cudaSuccess ? 1 : -1;
}

ADEPT_KTRACE_ATTACH(dg)

ADEPT_WAIT_LIMIT_SETTER(dg)

}  // namespace adept

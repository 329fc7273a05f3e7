// Grouped tcgen05 GEMM for sm_103a: C[M, N] = A[M, K] * B[N, K]^T per problem (bf16
// operands, both K-major; fp32 accumulation in tensor memory), one persistent launch
// over the tiles of every problem of the group, fused epilogues (epilogue.cuh).
//
// CTA = 6 warps:  warp 0 lane 0  TMA producer (A and B tiles, 128-byte swizzle)
//                 warp 1         tensor-memory allocator; lane 0 issues tcgen05.mma
//                 warps 2..5     epilogue: tcgen05.ld of the accumulator rows -> global
// Shared-memory ring of STAGES (A, B) k-blocks with full / empty mbarriers; two
// accumulator buffers in tensor memory so the epilogue of tile t overlaps the
// main loop of tile t+1.  Every mbarrier wait is bounded: on time-out the CTA sets
// ERRW_TIMEOUT in the device error word, stops, drains its MMAs and frees TMEM.
#define ADEPT_TU_ID 4
#include "gemm_tc.h"
#include "epilogue.cuh"
#include "tc_ptx.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <unordered_map>

namespace adept {

constexpr int TC_MAXG = 32;
constexpr int TC_BM = 128;
constexpr int TC_BK = 64;               // one 128-byte swizzle row of bf16
constexpr int TC_THREADS = 192;
constexpr int TC_SHORT_ROWS = 32;   // rows of the short-tile variants (3-D k-chunk boxes)
constexpr int TC_OUT_STAGE_BYTES = 4 * 32 * 32 * 4;   // epilogue TMA-store staging, one 32 x 32 fp32 chunk per warp
constexpr long long TC_TIMEOUT_CYCLES = 4000000000LL;   // ~2 s at 2 GHz

struct TcGroup {
  CUtensorMap ta;   // A: [rows, K] bf16, box 64 x 128
  CUtensorMap tb;   // B: [N, K] bf16, box 64 x BN
  CUtensorMap tout; // EPI_F32 output [rows, N] fp32, box 32 x 32, 128-byte swizzle (when tma_out)
  int tma_out;      // the epilogue stores 32 x 32 fp32 chunks by TMA instead of per-row stores
  DevRange rows;
  int N;
  int K;
  int gm;           // m-tiles per raster super-row (their A rows stay in L2 while n sweeps)
  int a_box;        // rows of A per TMA box: 128, or fewer when the whole problem is one short tile
                    // (the MMA still spans 128 rows; rows past the box are never stored)
  int m_lo, m_hi;   // live row-count gate: no tiles unless m_lo <= M and (m_hi == 0 or M <= m_hi)
  Epi epi;
};

template <int MAXG>
struct TcParams {
  TcGroup g[MAXG];
  int n_groups;
  unsigned* err;
};

// ---------------------------------------------------------------------------- PTX wrappers (tc_ptx.cuh)

// Instruction descriptor of kind::f16: D fp32, A and B bf16, both K-major, M = 128.
template <int BN>
__device__ __forceinline__ constexpr uint32_t idesc_bf16() {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(TC_BM >> 4) << 24);
}

#ifdef ADEPT_TC_TRACE
// Debug builds only (-DADEPT_TC_TRACE): clock64 timestamps of CTA 0's first tile, per
// launch, in a ring -- entry, TMEM ready, first TMA issued, first stage landed, last
// commit, accumulator seen by the epilogue, epilogue done, final barrier, TMEM freed.
__device__ long long g_tc_trace[256][16];
__device__ unsigned g_tc_launch;
#define TC_TRACE(k)                                                   \
  do {                                                                \
    if (blockIdx.x == 0 && tr_slot >= 0) g_tc_trace[tr_slot][k] = clock64(); \
  } while (0)
#else
#define TC_TRACE(k) \
  do {              \
  } while (0)
#endif

// ---------------------------------------------------------------------------- kernel
// KC > 1 (problems of at most TC_SHORT_ROWS rows, K a multiple of 64): a stage holds KC
// k-chunks loaded by one 3-D box per operand; the A chunks are packed a_box rows apart
// and the 128-row MMA of chunk c reads past its own rows into the next chunks (rows
// that are never stored), so the A region is one 128-row tile plus (KC-1) short tiles.
template <int BN, int STAGES, int MAXG, int KC>
__global__ void __launch_bounds__(TC_THREADS, 1) gemm_tc_kernel(const __grid_constant__ TcParams<MAXG> p) {
  KT_BEGIN();
  constexpr int A_BYTES = TC_BM * TC_BK * 2 + (KC - 1) * TC_SHORT_ROWS * TC_BK * 2;
  constexpr int B_BYTES = KC * BN * TC_BK * 2;
  constexpr uint32_t TMEM_COLS = 2 * BN;
  constexpr uint32_t IDESC = idesc_bf16<BN>();
  const long long wlim = wait_limit();   // the runtime wait limit, read once

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint8_t* sOut = smem + STAGES * (A_BYTES + B_BYTES);   // 4 x 4 KB: each epilogue warp's store chunk
  uint64_t* full = (uint64_t*)(sOut + TC_OUT_STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* accf = empty + STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  __shared__ int s_tile0[MAXG + 1];
  __shared__ int s_mbeg[MAXG], s_M[MAXG], s_tn[MAXG], s_tm[MAXG], s_gm[MAXG];
  __shared__ float s_bias[4][BN];   // epilogue: each warp's copy of the tile's bias columns

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ng = p.n_groups;
#ifdef ADEPT_TC_TRACE
  __shared__ int s_slot;
  if (threadIdx.x == 0) s_slot = blockIdx.x == 0 ? (int)(atomicAdd(&g_tc_launch, 1u) & 255u) : -1;
  __syncthreads();
  const int tr_slot = s_slot;
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    g_tc_trace[tr_slot][0] = clock64();
    g_tc_trace[tr_slot][9] = gridDim.x * 1000 + BN;
  }
#endif
  // Prologue that touches nothing an earlier kernel writes: barriers, the first group's
  // tensor maps (kernel parameters), the TMEM allocation.  Then wait for the preceding
  // kernels (programmatic dependent launch) and build the tile tables, which read row
  // counts those kernels produced.
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&p.g[0].ta) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&p.g[0].tb) : "memory");
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  pdl_wait();
  KT_WAITED();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int g = 0; g < ng; ++g) {
      const int b = p.g[g].rows.b();
      int M = max(0, p.g[g].rows.e() - b);
      if (M < p.g[g].m_lo || (p.g[g].m_hi > 0 && M > p.g[g].m_hi)) M = 0;
      const int tn = (p.g[g].N + BN - 1) / BN;
      s_mbeg[g] = b;
      s_M[g] = M;
      s_tn[g] = tn;
      s_tm[g] = (M + TC_BM - 1) / TC_BM;
      s_gm[g] = max(1, p.g[g].gm);
      s_tile0[g] = acc;
      acc += s_tm[g] * tn;
    }
    s_tile0[ng] = acc;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_launch_dependents();   // after the TMEM allocation: a dependent CTA cannot take it first
  const int total = s_tile0[ng];
  const uint32_t tmem = *tmem_slot;
  if ((int)blockIdx.x >= total) {
    // no tile for this CTA (uniform): give the tensor memory back and leave
    if (warp == 1) tmem_dealloc(tmem, TMEM_COLS);
    return;
  }
  if (threadIdx.x == 0 && ng > 1) {
    // the first tile's tensor maps, if they are not the first group's
    int g0 = 0;
    while (g0 + 1 < ng && (int)blockIdx.x >= s_tile0[g0 + 1]) ++g0;
    if (g0 > 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&p.g[g0].ta) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&p.g[g0].tb) : "memory");
    }
  }
  if (threadIdx.x == 0) TC_TRACE(1);

  // Tile order inside a problem: super-rows of gm m-tiles; within a super-row n is the
  // outer and m the inner index, so concurrently running CTAs share both the A rows of
  // the super-row and the weight slab of an n-block through L2.
  auto locate = [&](int t, int& g, int& mb, int& nb) {
    g = 0;
    while (g + 1 < ng && t >= s_tile0[g + 1]) ++g;
    const int local = t - s_tile0[g];
    const int gm = s_gm[g], tn = s_tn[g];
    const int sup = local / (gm * tn);
    const int rem = local - sup * gm * tn;
    const int rows = min(gm, s_tm[g] - sup * gm);
    nb = rem / rows;
    mb = sup * gm + rem % rows;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, last_par = 0;   // per stage: issued at least once / parity of its last issue
      int n_issued = 0;                    // slots are known free until the ring wraps once
      for (int t = blockIdx.x; t < total && !*abort_flag; t += gridDim.x) {
        int g, mb, nb;
        locate(t, g, mb, nb);
        const TcGroup& G = p.g[g];
        // per-tile values in registers: the asm "memory" clobbers below would otherwise make
        // every k-block reload them from parameter space
        const int nk = (G.K + TC_BK * KC - 1) / (TC_BK * KC);   // stages of KC k-chunks
        const int ya = s_mbeg[g] + mb * TC_BM, yb = nb * BN;
        const uint32_t tx_bytes = (uint32_t)(KC * (G.a_box + BN) * TC_BK * 2);
        const CUtensorMap* tma_a = &G.ta;
        const CUtensorMap* tma_b = &G.tb;
        for (int kb = 0; kb < nk; ++kb) {
          if (n_issued >= STAGES && !mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.err, wlim)) break;
          ++n_issued;
          mbar_expect_tx(&full[stage], tx_bytes);
          if (KC == 1) {
            tma_load_2d(tma_a, &full[stage], sA + stage * A_BYTES, kb * TC_BK, ya);
          } else {
            tma_load_3d(tma_a, &full[stage], sA + stage * A_BYTES, ya, kb * KC);
          }
          if (KC == 1) {
            tma_load_2d(tma_b, &full[stage], sB + stage * B_BYTES, kb * TC_BK, yb);
          } else {
            tma_load_3d(tma_b, &full[stage], sB + stage * B_BYTES, yb, kb * KC);
          }
          if (t == (int)blockIdx.x && kb == 0) TC_TRACE(2);
          issued |= 1u << stage;
          last_par = (last_par & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // every copy this thread issued has landed before the CTA may exit
      for (int s = 0; s < STAGES; ++s) {
        if (!(issued >> s & 1u)) continue;
        const uint32_t par = (last_par >> s) & 1u;
        const long long t0 = clock64();
        while (!mbar_try_wait(&full[s], par)) {
          if (clock64() - t0 > TC_TIMEOUT_CYCLES) {
            atomicOr(p.err, ERRW_TIMEOUT);
            break;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      int stage = 0, ab = 0;
      uint32_t phase = 0, aph = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
        int g, mb, nb;
        locate(t, g, mb, nb);
        const int nk = (p.g[g].K + TC_BK * KC - 1) / (TC_BK * KC);
        const uint32_t a_chunk = (uint32_t)(p.g[g].a_box * TC_BK * 2);   // bytes between A chunks
        if (!(ok = mbar_wait(&acce[ab], aph ^ 1, abort_flag, p.err, wlim))) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(ab * BN);
        for (int kb = 0; kb < nk; ++kb) {
          if (!(ok = mbar_wait(&full[stage], phase, abort_flag, p.err, wlim))) break;
          if (t == (int)blockIdx.x && kb == 0) TC_TRACE(3);

          tc_fence_after();
#pragma unroll
          for (int c = 0; c < KC; ++c) {
            const uint64_t ad = sdesc_sw128(smem_u32(sA + stage * A_BYTES) + c * a_chunk);
            const uint64_t bd = sdesc_sw128(smem_u32(sB + stage * B_BYTES) + c * (BN * TC_BK * 2));
#pragma unroll
            for (int k = 0; k < TC_BK / 16; ++k)
              umma_bf16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), IDESC, (kb | c | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        umma_commit(&accf[ab]);
        if (t == (int)blockIdx.x) TC_TRACE(4);
        ab ^= 1;
        if (ab == 0) aph ^= 1;
      }
      // drain: every MMA issued by this thread has completed before TMEM is freed
      umma_commit(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0)) {
        if (clock64() - t0 > TC_TIMEOUT_CYCLES) {
          atomicOr(p.err, ERRW_TIMEOUT);
          break;
        }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue warps 2..5
    const int q = warp & 3;                 // TMEM lane quarter this warp may access
    const int row_in_tile = q * 32 + lane;
    int ab = 0;
    uint32_t aph = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      int g, mb, nb;
      locate(t, g, mb, nb);
      const TcGroup& G = p.g[g];
      // the row's cache slot etc. do not depend on the accumulator: look them up first
      const int r = mb * TC_BM + row_in_tile;
      const bool valid = r < s_M[g];
      const int ra = s_mbeg[g] + r;
      EpiRow rr{-1, 0};
      if (valid) rr = epi_row(G.epi, ra);
      // the tile's bias columns, loaded once per warp (coalesced) while the accumulator fills,
      // instead of 32 broadcast loads per row chunk after it
      const float* bias = G.epi.bias;
      if (bias) {
        for (int c = lane; c < BN; c += 32) {
          const int col = nb * BN + c;
          s_bias[q][c] = col < G.N ? bias[col] : 0.f;
        }
        __syncwarp();
      }
      // one lane per warp polls the barrier (128 pollers would crowd the barrier unit the
      // producer and MMA threads need); the result is broadcast to the warp
      bool got = true;
      if (lane == 0) got = mbar_wait(&accf[ab], aph, abort_flag, p.err, wlim);
      got = __shfl_sync(0xffffffffu, got ? 1 : 0, 0) != 0;
      if (!got) break;   // warp-uniform: tcgen05.ld below is .sync.aligned
      if (t == (int)blockIdx.x && warp == 2 && lane == 0) TC_TRACE(5);
      tc_fence_after();
      const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN);
      if (G.tma_out) {
        // plain fp32 output: each 32 x 32 chunk goes to shared memory (row = lane, 16-byte
        // pieces in the 128-byte swizzle order) and leaves as one bulk tensor store, instead of
        // 32 row-strided 128-byte stores per warp instruction
        uint8_t* stg = sOut + q * 4096;
        const int y = s_mbeg[g] + mb * TC_BM + q * 32;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float v[32];
          tmem_ld32(tb + (uint32_t)c, v);
          const int c0 = nb * BN + c;
          if (c0 >= G.N) continue;   // warp-uniform
          if (bias) {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] += s_bias[q][c + j];
          }
          if (lane == 0) bulk_wait_read();   // the previous chunk's store has read the buffer
          __syncwarp();
          float4* row = reinterpret_cast<float4*>(stg + lane * 128);
#pragma unroll
          for (int k = 0; k < 8; ++k) row[k ^ (lane & 7)] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
          fence_async_shared();
          __syncwarp();
          if (lane == 0) tma_store_2d(&G.tout, stg, c0, y);
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float v[32];
          tmem_ld32(tb + (uint32_t)c, v);
          const int c0 = nb * BN + c;
          if (valid && c0 < G.N) epi_chunk32<bf16>(G.epi, ra, c0, G.N, v, rr, bias ? &s_bias[q][c] : nullptr);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (t == (int)blockIdx.x && warp == 2 && lane == 0) TC_TRACE(6);
      if (lane == 0) mbar_arrive(&acce[ab]);
      ab ^= 1;
      if (ab == 0) aph ^= 1;
    }
    if (lane == 0) bulk_wait_all();   // this warp's bulk stores are complete before the CTA ends
  }
  __syncthreads();
  if (threadIdx.x == 0) TC_TRACE(7);
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (threadIdx.x == 32) TC_TRACE(8);
}

// ---------------------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static int g_num_sms = 0;
static int g_cc_major = 0;

static void init_once() {
  static std::once_flag f;
  std::call_once(f, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    else
      cudaGetLastError();
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&g_cc_major, cudaDevAttrComputeCapabilityMajor, dev);
  });
}

bool tc_gemm_supported() {
  init_once();
  return g_encode != nullptr && g_cc_major == 10;
}

struct MapKey {
  const void* base;
  uint64_t inner, outer, row_bytes;
  uint32_t box;
  bool operator==(const MapKey& o) const {
    return base == o.base && inner == o.inner && outer == o.outer && row_bytes == o.row_bytes && box == o.box;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& k) const {
    size_t h = std::hash<const void*>()(k.base);
    h ^= std::hash<uint64_t>()(k.inner * 1315423911u + k.outer) + 0x9e3779b97f4a7c15ULL + (h << 6) + (h >> 2);
    h ^= std::hash<uint64_t>()(k.row_bytes * 2654435761u + k.box) + (h << 6) + (h >> 2);
    return h;
  }
};

// Tensor maps are encoded once per (address, extent, stride, box) and reused by later
// launches; a map depends on nothing else, so a reused address with the same extent
// maps the same way.
// Rows per A box: a problem whose rows fit one tile loads only a multiple of 8 rows that
// covers them (the TMA unit's cost grows with the rows of a box).
static int a_box_rows(int max_rows) {
  if (max_rows > 64) return TC_BM;
  int b = 8;
  while (b < max_rows) b *= 2;
  return b;
}

// m-tiles per raster super-row: their A rows (128 x K bf16 each) should take at most
// ~48 MiB of the 129 MiB L2, leaving room for the weight slabs and the output stream.
static int raster_gm(int K) {
  const long long per = 128LL * K * 2;
  return (int)std::max(1LL, std::min(64LL, (48LL << 20) / std::max(per, 1LL)));
}

static bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                     uint32_t box_outer) {
  if (((uintptr_t)base & 15) || (row_bytes & 15) || outer == 0 || inner == 0) return false;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  static std::mutex mu;
  const MapKey key{base, inner, outer, row_bytes, box_outer};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *m = it->second;
    return true;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {(cuuint32_t)TC_BK, box_outer};
  cuuint32_t estr[2] = {1, 1};
  if (g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  if (cache.size() > 65536) cache.clear();
  cache.emplace(key, *m);
  return true;
}

// fp32 output map of an EPI_F32 problem with a fixed row range: dims {N, rows}, box 32 x 32,
// 128-byte swizzle (the epilogue's staging order).  False when the output does not qualify.
static bool make_out_map(CUtensorMap* m, const GemmProblem& q) {
  if (q.epi.kind != EPI_F32 || q.rows.begin || q.rows.end || q.rows.count <= 0 || !q.epi.out_f32) return false;
  if (((uintptr_t)q.epi.out_f32 & 15) || (q.epi.ld_f32 & 3) || q.N <= 0) return false;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  static std::mutex mu;
  const uint64_t row_bytes = (uint64_t)q.epi.ld_f32 * 4;
  const MapKey key{q.epi.out_f32, (uint64_t)q.N, (uint64_t)q.rows.count, row_bytes, 32};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *m = it->second;
    return true;
  }
  cuuint64_t dims[2] = {(cuuint64_t)q.N, (cuuint64_t)q.rows.count};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  if (g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, q.epi.out_f32, dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  if (cache.size() > 65536) cache.clear();
  cache.emplace(key, *m);
  return true;
}

template <int BN, int STAGES, int MAXG, int KC = 1>
static int launch_bn(cudaStream_t st, const TcParams<MAXG>& prm, int grid) {
  constexpr size_t a_bytes = (size_t)TC_BM * TC_BK * 2 + (size_t)(KC - 1) * TC_SHORT_ROWS * TC_BK * 2;
  constexpr size_t b_bytes = (size_t)KC * BN * TC_BK * 2;
  constexpr size_t smem = (size_t)STAGES * (a_bytes + b_bytes) + TC_OUT_STAGE_BYTES + 1024 + 256;
  static_assert(smem <= 232448, "stage ring does not fit shared memory");
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(gemm_tc_kernel<BN, STAGES, MAXG, KC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    attr = true;
  }
  launch_k(gemm_tc_kernel<BN, STAGES, MAXG, KC>, grid, TC_THREADS, smem, st, prm);
  return 1;
}

// 3-D view {64, rows, K / 64} of a K-major matrix (strides: row, then 128 bytes per
// k-chunk), box {64, box_rows, kc}.
static bool encode_3d(CUtensorMap* m, const void* base, uint64_t K, uint64_t rows, uint64_t row_bytes,
                      uint32_t box_rows, uint32_t kc) {
  if (((uintptr_t)base & 15) || (row_bytes & 15) || rows == 0 || K == 0 || (K % TC_BK)) return false;
  // cached like the 2-D maps (a grouped fill encodes one map per layer on every call otherwise)
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  static std::mutex mu;
  const MapKey key{base, K, rows, row_bytes, box_rows | (kc << 16)};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *m = it->second;
    return true;
  }
  cuuint64_t dims[3] = {(cuuint64_t)TC_BK, rows, K / TC_BK};
  cuuint64_t strides[2] = {row_bytes, (cuuint64_t)TC_BK * 2};
  cuuint32_t box[3] = {(cuuint32_t)TC_BK, box_rows, kc};
  cuuint32_t estr[3] = {1, 1, 1};
  if (g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  if (cache.size() > 65536) cache.clear();
  cache.emplace(key, *m);
  return true;
}

bool tc_encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                  uint32_t box_outer) {
  init_once();
  if (!g_encode) return false;
  return make_map(m, base, inner, outer, row_bytes, box_outer);
}

bool tc_encode_weight_3d(CUtensorMap* m, const void* base, int K, int rows, size_t row_bytes, int box_rows, int kc) {
  init_once();
  if (!g_encode) return false;
  return encode_3d(m, base, (uint64_t)K, (uint64_t)rows, (uint64_t)row_bytes, (uint32_t)box_rows, (uint32_t)kc);
}

// Tile width for row bounds max_rows: the widest that still gives every SM a tile; *tiles
// the tile count at that width.
static int pick_bn(const GemmProblem* probs, int n_probs, const int* max_rows, long long* tiles_out) {
  long long tiles[4] = {0, 0, 0, 0};
  const int bns[4] = {256, 128, 64, 32};
  for (int i = 0; i < n_probs; ++i) {
    const long long tm = (max_rows[i] + TC_BM - 1) / TC_BM;
    for (int k = 0; k < 4; ++k) tiles[k] += tm * ((probs[i].N + bns[k] - 1) / bns[k]);
  }
  int pick = 3;
  for (int k = 0; k < 4; ++k)
    if (tiles[k] >= g_num_sms) {
      pick = k;
      break;
    }
  // wave quantisation: the next narrower width (down to 128) when its whole waves of tiles take
  // at least 10 % less work per SM (e.g. 512 tiles of 256 are 4 waves of 256 columns on 152 SMs,
  // 1024 tiles of 128 are 7 waves of 128)
  if (pick < 3 && bns[pick + 1] >= 128) {
    const long long w0 = (tiles[pick] + g_num_sms - 1) / g_num_sms * bns[pick];
    const long long w1 = (tiles[pick + 1] + g_num_sms - 1) / g_num_sms * bns[pick + 1];
    if (w1 * 10 <= w0 * 9) ++pick;
  }
  *tiles_out = tiles[pick];
  return bns[pick];
}

// A prepared launch: parameters (tensor maps encoded), tile width, k-chunks per stage, grid.
template <int MAXG>
struct TcPrepared {
  TcParams<MAXG> prm;
  int BN, KC, grid;
};

// Fills `L` for problems with row bounds max_rows and the live row-count gate [m_lo, m_hi]
// (m_hi = 0: none); tile width force_bn, or (0) pick_bn's.  -1 when a tensor map cannot be
// encoded (nothing launched).
template <int MAXG>
static int prepare_grouped(TcPrepared<MAXG>& L, const GemmProblem* probs, int n_probs, const int* max_rows,
                           unsigned* err_word, int m_lo, int m_hi, int force_bn = 0) {
  long long n_tiles = 0;
  int BN = pick_bn(probs, n_probs, max_rows, &n_tiles);
  if (force_bn) {
    BN = force_bn;
    n_tiles = 0;
    for (int i = 0; i < n_probs; ++i)
      n_tiles += (long long)((max_rows[i] + TC_BM - 1) / TC_BM) * ((probs[i].N + BN - 1) / BN);
  }
  // short problems (every group one tile of at most TC_SHORT_ROWS rows, K in whole 64-chunks)
  // take the 3-D box variant: one TMA instruction per operand carries KC k-chunks
  bool short_rows = true;
  for (int i = 0; i < n_probs; ++i)
    short_rows &= max_rows[i] <= TC_SHORT_ROWS && probs[i].K % TC_BK == 0;
  const int KC = short_rows ? (BN == 256 ? 2 : 4) : 1;
  TcParams<MAXG>& prm = L.prm;
  memset(&prm, 0, sizeof prm);
  prm.n_groups = n_probs;
  prm.err = err_word;
  for (int i = 0; i < n_probs; ++i) {
    const GemmProblem& q = probs[i];
    TcGroup& G = prm.g[i];
    G.m_lo = m_lo;
    G.m_hi = m_hi;
    G.a_box = a_box_rows(max_rows[i]);
    if (KC > 1) {
      if (!encode_3d(&G.ta, q.A, (uint64_t)q.K, (uint64_t)q.a_rows, (uint64_t)q.lda * 2, (uint32_t)G.a_box,
                     (uint32_t)KC))
        return -1;
      if (!encode_3d(&G.tb, q.B, (uint64_t)q.K, (uint64_t)q.N, (uint64_t)q.ldb * 2, (uint32_t)BN, (uint32_t)KC))
        return -1;
    } else {
      if (!make_map(&G.ta, q.A, (uint64_t)q.K, (uint64_t)q.a_rows, (uint64_t)q.lda * 2, (uint32_t)G.a_box))
        return -1;
      if (!make_map(&G.tb, q.B, (uint64_t)q.K, (uint64_t)q.N, (uint64_t)q.ldb * 2, (uint32_t)BN)) return -1;
    }
    G.rows = q.rows;
    G.N = q.N;
    G.K = q.K;
    G.gm = raster_gm(q.K);
    G.epi = q.epi;
    G.tma_out = make_out_map(&G.tout, q) ? 1 : 0;
  }
  L.BN = BN;
  L.KC = KC;
  L.grid = (int)std::min<long long>(n_tiles, (long long)g_num_sms);
  return 0;
}

template <int MAXG>
static int launch_prepared(cudaStream_t st, const TcPrepared<MAXG>& L) {
  const int grid = L.grid;
  if (grid <= 0) return 0;
  if (L.KC > 1) {
    switch (L.BN) {
      case 256: return launch_bn<256, 2, MAXG, 2>(st, L.prm, grid);
      case 128: return launch_bn<128, 2, MAXG, 4>(st, L.prm, grid);
      case 64: return launch_bn<64, 3, MAXG, 4>(st, L.prm, grid);
      default: return launch_bn<32, 4, MAXG, 4>(st, L.prm, grid);
    }
  }
  switch (L.BN) {
    case 256: return launch_bn<256, 4, MAXG>(st, L.prm, grid);
    case 128: return launch_bn<128, 6, MAXG>(st, L.prm, grid);
    case 64: return launch_bn<64, 8, MAXG>(st, L.prm, grid);
    default: return launch_bn<32, 10, MAXG>(st, L.prm, grid);
  }
}

template <int MAXG>
static int launch_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows,
                          unsigned* err_word) {
  // kept off the stack; one per host thread, so threads driving different models do not share it
  thread_local TcPrepared<MAXG> L;
  if (prepare_grouped(L, probs, n_probs, max_rows, err_word, 0, 0) < 0) return -1;
  return launch_prepared(st, L);
}

// One problem whose live row count is on the device and usually far below its bound (the
// prompt pass's exiting rows, flagged split_live): the host knows only the bound, whose tile
// width can leave most SMs idle for the live count.  Two launches then share the problem: one
// with the next narrower tiles for live counts up to m_split rows, the most row tiles that
// width still fits in one wave (there each CTA loads (128 + BN) x K per tile instead of
// (128 + 2 BN) x K, and twice the SMs pull), and the bound's launch for larger counts.  Each
// finds no tiles when the count is outside its range, so exactly one of them runs the
// product.  Both are prepared before either is launched.  Returns the launch count, or -1 when
// the split does not apply.
// The plan of that split for N columns and the row bound max_rows on `sms` SMs: the bound's
// tile width (pick_bn's choice for one problem), the next narrower width, and m_split; false
// when the split does not apply (one row tile, the narrowest width already, or one row tile of
// the narrower width does not fit in one wave).
static bool split_plan(int N, int max_rows, int sms, int* bn_wide, int* bn_narrow, int* m_split) {
  if (max_rows <= TC_BM || N <= 0 || sms <= 0) return false;
  const long long tm = (max_rows + TC_BM - 1) / TC_BM;
  const int bns[4] = {256, 128, 64, 32};
  int w = 32;
  for (int k = 0; k < 4; ++k)
    if (tm * ((N + bns[k] - 1) / bns[k]) >= sms) {
      w = bns[k];
      break;
    }
  if (w <= 32) return false;
  const int nb = w / 2;
  const long long row_tiles = sms / ((N + nb - 1) / nb);
  if (row_tiles < 1) return false;
  *bn_wide = w;
  *bn_narrow = nb;
  *m_split = (int)std::min<long long>(row_tiles * TC_BM, (long long)max_rows - 1);
  return true;
}

static int launch_split_live_rows(cudaStream_t st, const GemmProblem& q, int max_rows, unsigned* err_word) {
  if (!q.split_live || !(q.rows.begin || q.rows.end)) return -1;
  int bn_wide = 0, bn_narrow = 0, m_split = 0;
  if (!split_plan(q.N, max_rows, g_num_sms, &bn_wide, &bn_narrow, &m_split)) return -1;
  thread_local TcPrepared<2> narrow, wide;
  if (prepare_grouped(narrow, &q, 1, &m_split, err_word, 0, m_split, bn_narrow) < 0) return -1;
  if (prepare_grouped(wide, &q, 1, &max_rows, err_word, m_split + 1, 0) < 0) return -1;
  return launch_prepared(st, narrow) + launch_prepared(st, wide);
}

int tc_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows, unsigned* err_word) {
  init_once();
  if (n_probs <= 0) return 0;
  if (n_probs > TC_MAXG) return -1;
  // the cache / SwiGLU epilogues work on whole 32-column chunks
  for (int i = 0; i < n_probs; ++i) {
    const GemmProblem& q = probs[i];
    if (q.K % 8 || q.lda % 8 || q.ldb % 8 || q.a_rows <= 0) return -1;
    if ((q.epi.kind == EPI_QKV || q.epi.kind == EPI_KV || q.epi.kind == EPI_SWIGLU) && (q.N % 32)) return -1;
  }
  if (n_probs == 1) {
    const int nl = launch_split_live_rows(st, probs[0], max_rows[0], err_word);
    if (nl >= 0) return nl;
  }
  // small launches carry a small parameter block (cheaper to launch)
  if (n_probs <= 2) return launch_grouped<2>(st, probs, n_probs, max_rows, err_word);
  return launch_grouped<TC_MAXG>(st, probs, n_probs, max_rows, err_word);
}

// Same launch as tc_gemm_grouped, for callers that must not allocate: the tensor maps are
// encoded into the launch parameters on every call (no map cache, no host heap use).
int tc_gemm_grouped_nocache(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows,
                            unsigned* err_word) {
  init_once();
  if (n_probs <= 0) return 0;
  if (n_probs > TC_MAXG || !g_encode) return -1;
  long long tiles[4] = {0, 0, 0, 0};
  const int bns[4] = {256, 128, 64, 32};
  for (int i = 0; i < n_probs; ++i) {
    const GemmProblem& q = probs[i];
    if (q.K % 8 || q.lda % 8 || q.ldb % 8 || q.a_rows <= 0) return -1;
    if ((q.epi.kind == EPI_QKV || q.epi.kind == EPI_KV || q.epi.kind == EPI_SWIGLU) && (q.N % 32)) return -1;
    const long long tm = (max_rows[i] + TC_BM - 1) / TC_BM;
    for (int k = 0; k < 4; ++k) tiles[k] += tm * ((q.N + bns[k] - 1) / bns[k]);
  }
  int pick = 3;
  for (int k = 0; k < 4; ++k)
    if (tiles[k] >= g_num_sms) {
      pick = k;
      break;
    }
  const int BN = bns[pick];
  thread_local TcParams<TC_MAXG> prm;  // per host thread, not on the heap
  memset(&prm, 0, sizeof prm);
  prm.n_groups = n_probs;
  prm.err = err_word;
  auto encode = [&](CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                    uint32_t box_outer) {
    if (((uintptr_t)base & 15) || (row_bytes & 15) || outer == 0 || inner == 0) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {(cuuint32_t)TC_BK, box_outer};
    cuuint32_t estr[2] = {1, 1};
    return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  };
  for (int i = 0; i < n_probs; ++i) {
    const GemmProblem& q = probs[i];
    TcGroup& G = prm.g[i];
    G.a_box = a_box_rows(max_rows[i]);
    if (!encode(&G.ta, q.A, (uint64_t)q.K, (uint64_t)q.a_rows, (uint64_t)q.lda * 2, (uint32_t)G.a_box)) return -1;
    if (!encode(&G.tb, q.B, (uint64_t)q.K, (uint64_t)q.N, (uint64_t)q.ldb * 2, (uint32_t)BN)) return -1;
    G.rows = q.rows;
    G.N = q.N;
    G.K = q.K;
    G.gm = raster_gm(q.K);
    G.epi = q.epi;
  }
  const int grid = (int)std::min<long long>(tiles[pick], (long long)g_num_sms);
  if (grid <= 0) return 0;
  switch (BN) {
    case 256: return launch_bn<256, 4, TC_MAXG>(st, prm, grid);
    case 128: return launch_bn<128, 6, TC_MAXG>(st, prm, grid);
    case 64: return launch_bn<64, 8, TC_MAXG>(st, prm, grid);
    default: return launch_bn<32, 10, TC_MAXG>(st, prm, grid);
  }
}

ADEPT_KTRACE_ATTACH(tc)

ADEPT_WAIT_LIMIT_SETTER(tc)

}  // namespace adept

// Host-side check of the live-row split plan (no device work): returns 1 and {bound's tile
// width, narrower width, m_split} in out3, or 0 when the split does not apply.
extern "C" __attribute__((visibility("default"))) int adept_debug_tc_split_plan(int N, int max_rows, int sms,
                                                                                 int* out3) {
  int a = 0, b = 0, c = 0;
  if (!adept::split_plan(N, max_rows, sms, &a, &b, &c)) return 0;
  out3[0] = a;
  out3[1] = b;
  out3[2] = c;
  return 1;
}

#ifdef ADEPT_TC_TRACE
extern "C" __attribute__((visibility("default"))) int adept_debug_tc_trace(long long* out, unsigned* n_launches) {
  if (cudaMemcpyFromSymbol(out, adept::g_tc_trace, sizeof(long long) * 256 * 16) != cudaSuccess) return 1;
  if (cudaMemcpyFromSymbol(n_launches, adept::g_tc_launch, sizeof(unsigned)) != cudaSuccess) return 1;
  return 0;
}
#endif

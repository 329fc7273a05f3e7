// Skinny GEMM for passes of at most 32 token rows (generation steps, output heads):
// C[M, N] = A[M, K] * W[N, K]^T with M <= 32.  Such a GEMM is a stream over the weights,
// so the kernel is shaped for bandwidth: the weights are the tensor-core M operand
// (64 output features per CTA, 16 per warp, mma.sync m16n8k16 bf16 with the tokens as
// the n8 blocks), K is split across CTAs until the grid covers the GPU twice, and a
// 4-stage cp.async ring streams 64 x 64 weight tiles.  Each split writes its partial
// tile to a workspace slot; the last CTA of a tile (an arrival counter) sums the slots
// in split order -- the result does not depend on timing -- and applies the fused
// epilogue (epilogue.cuh) on 32-column chunks, then resets the counter.
#include "gemm_skinny.h"
#include "epilogue.cuh"

#include <algorithm>
#include <cstring>

namespace adept {

constexpr int SK_BN = 64;       // output features per tile
constexpr int SK_BK = 64;       // k per stage
constexpr int SK_STAGES = 4;
constexpr int SK_LDS = SK_BK + 8;   // padded smem rows (bf16 elements)
constexpr int SK_THREADS = 128;
constexpr int SK_SLOT = SK_BN * SKINNY_MAX_M;   // floats per partial tile

struct SkGroup {
  const bf16* A;
  const bf16* W;
  int lda, ldw;
  DevRange rows;
  int N, K;
  int tiles, splits, kchunk;
  int cta0;    // first CTA of this group
  int tile0;   // first global tile (counter / slot index)
  Epi epi;
};

template <int MAXG>
struct SkParams {
  SkGroup g[MAXG];
  int n_groups;
  float* ws;
  int* counters;
};

__device__ __forceinline__ void sk_cp16(void* smem, const void* gmem, bool valid) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(smem);
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(a), "l"(gmem), "r"(n) : "memory");
}
__device__ __forceinline__ void sk_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void sk_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void sk_ldsm_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3, const void* p) {
  const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void sk_mma(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int MAXG, int MB>   // MB: 8-token blocks (1..4)
__global__ void __launch_bounds__(SK_THREADS) gemm_skinny_kernel(const __grid_constant__ SkParams<MAXG> p) {
  PDL_ENTRY();
  extern __shared__ __align__(16) uint8_t sk_smem[];
  bf16* sW = reinterpret_cast<bf16*>(sk_smem);                          // [STAGES][64][LDS]
  bf16* sA = sW + SK_STAGES * SK_BN * SK_LDS;                           // [STAGES][32][LDS]
  float* sC = reinterpret_cast<float*>(sA + SK_STAGES * SKINNY_MAX_M * SK_LDS);   // [32][64 + 4]
  __shared__ int s_last;

  // which group / tile / split
  int gi = 0;
  while (gi + 1 < p.n_groups && (int)blockIdx.x >= p.g[gi + 1].cta0) ++gi;
  const SkGroup& G = p.g[gi];
  const int local = blockIdx.x - G.cta0;
  const int tile = local / G.splits, split = local % G.splits;
  const int rb = G.rows.b();
  const int M = min(G.rows.e() - rb, SKINNY_MAX_M);
  if (M <= 0) return;  // same for every CTA of the group: no counter is touched
  const int f0 = tile * SK_BN;
  const int k_lo = split * G.kchunk;
  const int k_hi = min(G.K, k_lo + G.kchunk);
  const int nkb = k_hi > k_lo ? (k_hi - k_lo + SK_BK - 1) / SK_BK : 0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  auto load_stage = [&](int s, int kb) {
    const int k0 = k_lo + kb * SK_BK;
    bf16* w = sW + s * SK_BN * SK_LDS;
    bf16* a = sA + s * SKINNY_MAX_M * SK_LDS;
    for (int c = tid; c < SK_BN * (SK_BK / 8); c += SK_THREADS) {
      const int r = c >> 3, kc = (c & 7) * 8;
      const int f = f0 + r, k = k0 + kc;
      const bool ok = f < G.N && k < k_hi;
      sk_cp16(w + r * SK_LDS + kc, ok ? (const void*)(G.W + (size_t)f * G.ldw + k) : (const void*)G.W, ok);
    }
    for (int c = tid; c < MB * 8 * (SK_BK / 8); c += SK_THREADS) {
      const int r = c >> 3, kc = (c & 7) * 8;
      const int k = k0 + kc;
      const bool ok = r < M && k < k_hi;
      sk_cp16(a + r * SK_LDS + kc, ok ? (const void*)(G.A + (size_t)(rb + r) * G.lda + k) : (const void*)G.A, ok);
    }
  };

  float acc[MB][4];
#pragma unroll
  for (int j = 0; j < MB; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

#pragma unroll
  for (int s = 0; s < SK_STAGES - 1; ++s) {
    if (s < nkb) load_stage(s, s);
    sk_commit();
  }
  for (int kb = 0; kb < nkb; ++kb) {
    sk_wait<SK_STAGES - 2>();
    __syncthreads();
    {
      const int nx = kb + SK_STAGES - 1;
      if (nx < nkb) load_stage(nx % SK_STAGES, nx);
      sk_commit();
    }
    const int s = kb % SK_STAGES;
    const bf16* w = sW + s * SK_BN * SK_LDS;
    const bf16* a = sA + s * SKINNY_MAX_M * SK_LDS;
#pragma unroll
    for (int kk = 0; kk < SK_BK / 16; ++kk) {
      uint32_t af[4];
      {
        const int mi = lane >> 3;
        const int row = warp * 16 + (mi & 1) * 8 + (lane & 7);
        const int col = kk * 16 + (mi >> 1) * 8;
        sk_ldsm_x4(af[0], af[1], af[2], af[3], w + row * SK_LDS + col);
      }
#pragma unroll
      for (int jp = 0; jp < (MB + 1) / 2; ++jp) {  // two 8-token blocks per ldmatrix
        const int mi = lane >> 3;
        const int tok = jp * 16 + (mi >> 1) * 8 + (lane & 7);
        const int col = kk * 16 + (mi & 1) * 8;
        uint32_t b0, b1, b2, b3;
        sk_ldsm_x4(b0, b1, b2, b3, a + tok * SK_LDS + col);
        sk_mma(acc[2 * jp], af, b0, b1);
        if (2 * jp + 1 < MB) sk_mma(acc[2 * jp + 1], af, b2, b3);
      }
    }
  }
  sk_wait<0>();

  // partial tile -> workspace slot [feature][token]
  const int g = lane >> 2, t4 = lane & 3;
  float* slot = p.ws + ((size_t)(G.tile0 + tile) * G.splits + split) * SK_SLOT;
#pragma unroll
  for (int j = 0; j < MB; ++j) {
    const int fr = warp * 16 + g, tk = j * 8 + 2 * t4;
    slot[(fr)*SKINNY_MAX_M + tk] = acc[j][0];
    slot[(fr)*SKINNY_MAX_M + tk + 1] = acc[j][1];
    slot[(fr + 8) * SKINNY_MAX_M + tk] = acc[j][2];
    slot[(fr + 8) * SKINNY_MAX_M + tk + 1] = acc[j][3];
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int prev = atomicAdd(&p.counters[G.tile0 + tile], 1);
    s_last = (prev == G.splits - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // last CTA of the tile: sum the splits in order, transpose to [token][feature]
  const float* base = p.ws + (size_t)(G.tile0 + tile) * G.splits * SK_SLOT;
  for (int e = tid; e < SK_BN * MB * 8; e += SK_THREADS) {
    const int fr = e / (MB * 8), tk = e % (MB * 8);
    float v = 0.f;
    for (int s = 0; s < G.splits; ++s) v += __ldcg(base + (size_t)s * SK_SLOT + fr * SKINNY_MAX_M + tk);
    sC[tk * (SK_BN + 4) + fr] = v;
  }
  __syncthreads();
  if (tid == 0) p.counters[G.tile0 + tile] = 0;
  // epilogue: (token, 32-column chunk) items
  for (int it = tid; it < M * (SK_BN / 32); it += SK_THREADS) {
    const int tk = it / (SK_BN / 32), ch = it % (SK_BN / 32);
    const int c0 = f0 + ch * 32;
    if (c0 >= G.N) continue;
    float v[32];
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) v[jj] = sC[tk * (SK_BN + 4) + ch * 32 + jj];
    const int ra = rb + tk;
    const EpiRow rr = epi_row(G.epi, ra);
    epi_chunk32<bf16>(G.epi, ra, c0, G.N, v, rr);
  }
}

static int g_sms = 0;

template <int MAXG, int MB>
static void launch_mb(cudaStream_t st, const SkParams<MAXG>& prm, int grid) {
  constexpr int smem = (SK_STAGES * (SK_BN + SKINNY_MAX_M) * SK_LDS) * 2 + SKINNY_MAX_M * (SK_BN + 4) * 4;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(gemm_skinny_kernel<MAXG, MB>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    attr = true;
  }
  launch_k(gemm_skinny_kernel<MAXG, MB>, grid, SK_THREADS, smem, st, prm);
}

template <int MAXG>
static int launch_groups(cudaStream_t st, const GemmProblem* probs, int n, int max_m, float* ws, size_t ws_floats,
                         int* counters, int n_counters) {
  static SkParams<MAXG> prm;
  memset(&prm, 0, sizeof prm);
  prm.n_groups = n;
  prm.ws = ws;
  prm.counters = counters;
  int tiles_total = 0;
  for (int i = 0; i < n; ++i) tiles_total += (probs[i].N + SK_BN - 1) / SK_BN;
  // splits: enough CTAs to cover the GPU twice, at least 128 k per split
  int cta = 0, tile0 = 0;
  size_t slots = 0;
  for (int i = 0; i < n; ++i) {
    const GemmProblem& q = probs[i];
    SkGroup& G = prm.g[i];
    G.A = (const bf16*)q.A;
    G.W = (const bf16*)q.B;
    G.lda = q.lda;
    G.ldw = q.ldb;
    G.rows = q.rows;
    G.N = q.N;
    G.K = q.K;
    G.tiles = (q.N + SK_BN - 1) / SK_BN;
    int s = std::max(1, (2 * g_sms + tiles_total - 1) / std::max(tiles_total, 1));
    s = std::min(s, std::max(1, q.K / 128));
    int kchunk = (q.K + s - 1) / s;
    kchunk = ((kchunk + SK_BK - 1) / SK_BK) * SK_BK;
    s = (q.K + kchunk - 1) / kchunk;
    G.splits = s;
    G.kchunk = kchunk;
    G.cta0 = cta;
    G.tile0 = tile0;
    G.epi = q.epi;
    cta += G.tiles * s;
    tile0 += G.tiles;
    slots += (size_t)G.tiles * s;
  }
  if (tile0 > n_counters || slots * SK_SLOT > ws_floats) return -1;
  if (cta == 0) return 0;
  const int mb = (max_m + 7) / 8;
  switch (mb) {
    case 1: launch_mb<MAXG, 1>(st, prm, cta); break;
    case 2: launch_mb<MAXG, 2>(st, prm, cta); break;
    case 3: launch_mb<MAXG, 3>(st, prm, cta); break;
    default: launch_mb<MAXG, 4>(st, prm, cta); break;
  }
  return 1;
}

int skinny_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows, float* ws,
                        size_t ws_floats, int* counters, int n_counters) {
  if (n_probs <= 0) return 0;
  if (n_probs > 32) return -1;
  if (!g_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
  }
  int max_m = 0;
  for (int i = 0; i < n_probs; ++i) {
    const GemmProblem& q = probs[i];
    if (max_rows[i] > SKINNY_MAX_M) return -1;
    if (q.K % 8 || q.lda % 8 || q.ldb % 8 || ((uintptr_t)q.A & 15) || ((uintptr_t)q.B & 15)) return -1;
    if ((q.epi.kind == EPI_QKV || q.epi.kind == EPI_KV || q.epi.kind == EPI_SWIGLU) && (q.N % 32)) return -1;
    max_m = std::max(max_m, max_rows[i]);
  }
  if (n_probs <= 2) return launch_groups<2>(st, probs, n_probs, max_m, ws, ws_floats, counters, n_counters);
  return launch_groups<32>(st, probs, n_probs, max_m, ws, ws_floats, counters, n_counters);
}

}  // namespace adept

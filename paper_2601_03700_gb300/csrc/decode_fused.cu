// Persistent generation-step kernel for small batches of a bf16 decoder: the whole
// early-exit step (Sec. 4, App. I) in ONE cooperative launch of one CTA per SM --
// every computed layer (standardised input -> QKV + RoPE + cache write, attention over
// the paged cache, O + residual, standardised input -> FFN, down + residual, the exit
// test with active-token compaction), then the HSM of the exited tokens (Sec. 4.2,
// Table S1), their skipped-layer K/V fills (Sec. 4.3) and the LM head with greedy argmax.
//
// A generation step of a few tokens is weight streaming plus ~100 dependent steps.  As
// separate launches each step pays launch, prologue and pipeline-fill latency.  Here the
// steps are phases separated by grid barriers, and a producer warp per CTA streams the
// CTA's slices of the weight matrices through a shared-memory ring with TMA on its own
// schedule: the weights of the next projection are in flight while the attention, the
// exit test or a barrier of the previous phase runs.
//
// CTA = 8 warps.  Warp 7 lane 0: TMA producer.  Warps 0..6: consumers (operand staging,
// attention, exit test, HSM row steps, epilogues); warps 0..3 also issue the mma.sync
// contractions.  A contraction is computed as C^T = W X^T: weight rows are the MMA's M
// side (32 per tile, two m16 tiles), the <= 16 token rows its N side (n8 groups), so no
// tensor-core work is spent on padding rows of a 128-row tile.  The unit of work is one
// stage of 32 weight rows x 256 k (16 KiB, one 3-D TMA box of four swizzled 64-k
// chunks); each CTA takes a contiguous range of a phase's units (stream-K), and a tile
// split between CTAs is summed in a fixed order by its last contributor, so results do
// not depend on timing.  Every wait is bounded: on time-out the CTA sets ERRW_TIMEOUT,
// every role leaves its loop, the producer waits for its copies in flight, and the
// other CTAs leave their barrier waits when they see the error bit.
#include "decode_fused.h"
#include "adept.h"
#include "epilogue.cuh"
#include "gemm_tc.h"
#include "kernels.h"

#include <cuda.h>

#include <algorithm>
#include <mutex>
#include <cmath>
#include <cstring>
#include <vector>

namespace adept {
namespace {

constexpr int kThreads = 256;
constexpr int kCons = 224;           // consumer threads (warps 0..6)
constexpr int kConsWarps = 7;
constexpr int kMmaWarps = 4;
constexpr int kTN = 32;              // weight rows (output columns) per tile
constexpr int kKC = 4;               // 64-wide k chunks per stage
constexpr int kSK = kKC * 64;        // k per stage
constexpr int kStageBytes = kTN * kSK * 2;
constexpr int kMaxB = DF_MAX_BATCH;
constexpr int kAttnMaxSplit = 64;
constexpr int kMaxProbs = DF_MAX_LAYERS + 1;
constexpr int kStashProbs = 4;     // epilogue descriptors of a CTA's tiles staged per phase
constexpr int kStashTiles = 16;    // bias slices staged per phase
constexpr int kStashResid = 2;     // residual slices staged per phase
constexpr int kRopeRows = 4;       // tokens whose RoPE rows are staged per step
constexpr long long kTimeout = 4000000000LL;   // ~2 s at 2 GHz

#ifdef ADEPT_DF_TRACE
// Debug builds only (-DADEPT_DF_TRACE): clock64 cycles per activity, accumulated by
// consumer thread 0 (an MMA lane) and the producer thread of CTA 0 and of CTA grid/2.
enum : int {
  TB_TOTAL = 0, TB_EMBED, TB_SYNC, TB_LOADX, TB_MMA, TB_FULLWAIT, TB_REDUCE, TB_EPI, TB_FIXUP, TB_ATTN, TB_EXIT,
  TB_HSMOUT, TB_ARGMAX, TB_NSYNC, TB_PEMPTY, TB_PFLAG, TB_FREEWAIT, TB_NFULL, TB_NSPLIT, TB_SX_LOAD, TB_SX_MEAN,
  TB_SX_VAR, TB_SX_OUT, TB_N
};
__device__ unsigned long long g_df_prof[2][32];
__device__ unsigned long long g_df_work[256][16];
enum : int { WK_EMBED = 0, WK_QKV, WK_ATTN, WK_O, WK_UP, WK_DOWN, WK_EXIT, WK_FINAL, WK_H1, WK_H2, WK_H3, WK_H4,
             WK_OUT, WK_FILLHEAD };
#define DF_PH(k)                         \
  do {                                   \
    if (threadIdx.x == 0) sh.cur = (k);  \
  } while (0)
#define DF_CLK(v) const long long v = clock64()
#define DF_C(b, t0)                                   \
  do {                                                \
    if (threadIdx.x == 0) sh.pc[b] += clock64() - (t0); \
  } while (0)
#define DF_P(b, t0) sh.pc[b] += clock64() - (t0)
#define DF_E(b, t0)                                      \
  do {                                                   \
    if (threadIdx.x == 128) sh.pc[b] += clock64() - (t0); \
  } while (0)
#else
#define DF_E(b, t0) \
  do {              \
  } while (0)
#define DF_CLK(v)
#define DF_C(b, t0) \
  do {              \
  } while (0)
#define DF_P(b, t0) \
  do {              \
  } while (0)
#define DF_PH(k) \
  do {           \
  } while (0)
#endif

#ifdef ADEPT_DF_TRACE
// Debug builds: an access about to leave its buffer records (code, detail) once, sets
// ERRW_CONFIG and is skipped.
#define DF_CHECK(P, cond, code, detail)                                        \
  ((cond) ? true                                                              \
          : (atomicOr((P).err, ERRW_CONFIG), atomicCAS((P).dbg, 0u, (unsigned)(code)) == 0u \
                                                    ? (void)atomicExch((P).dbg + 1, (unsigned)(detail)) \
                                                    : (void)0,                                      \
             false))
#else
#define DF_CHECK(P, cond, code, detail) true
#endif

enum PhaseKind : int { PH_QKV = 0, PH_O, PH_UP, PH_DOWN, PH_H1, PH_H2, PH_H3, PH_H4, PH_FILLHEAD };

struct DfLayerDev {
  CUtensorMap m_qkv, m_o, m_up, m_down, m_kv;   // 3-D weight views {64, rows, K/64}, box {64, 32, 4}
  Epi e_qkv, e_o, e_up, e_down, e_kv;
};

struct DfPlan {
  CUtensorMap m_h[4];
  CUtensorMap m_head;
  Epi e_h[4];
  Epi e_head;
  const DfLayerDev* L;
  int N, D, Dq, Dkv, H, Hkv, dh, F, up_rows, V, m1, m2, family, norm_mode, nqkv;
  float eps, hsm_eps;
  int seq_cap, max_pos;
  const bf16* tok_emb;
  const bf16* pos_emb;
  const float *hsm_g0, *hsm_conv, *hsm_g1, *hsm_g2;
  KVCacheView cache;
  float* X_in[2];
  float* X_out;
  float* I[2];
  int* row_tok[2];
  int *tok_seq, *tok_pos, *seq_len, *ctr;
  unsigned* err;
  bf16 *q, *att, *hbuf, *xfill, *h1t, *h2t;
  float *hsm_s, *hsm_prev, *hsm_I, *final_, *c0f, *h1f, *h3f, *h5f;
  int* exit_tok;
  long long lstride;     // cache elements between layers
  long long pool_elems;  // elements of each of the K and V pools
  int bt_shift;          // log2(block_tokens) when a power of two, else -1
  const float2* rope_table;
  unsigned* dbg;         // debug builds: first failed self-check (code, detail)
  float* attn_ws;        // [rows * H * kAttnMaxSplit][dh + 2]
  unsigned* attn_cnt;    // [kMaxB * H]
  float* amax_v;         // [grid][kMaxB]
  int* amax_i;
  unsigned* amax_cnt;
  unsigned* bar;         // [0] arrivals, [1] generation
};

struct DfCall {
  const DfPlan* P;
  const int* tokens;
  const int* forced;
  float delta;
  int B;
  int identity;
  int* exit_out;
  float* sim_out;
  int* next_out;
  int ring;
  int x_bytes;
  int attn_chunk;
  int attn_nsplit;
  int rb;           // token stride of the reduction buffers (8 or 16)
  long long lstride;       // cache elements between layers
  int pos[DF_MAX_BATCH];   // position of each sequence's new token
};

struct DfProb {
  const CUtensorMap* map;
  const Epi* epi;
  int N, K, tiles, S, xblk, rows, tile0;
};

struct DfPhase {
  DfProb p[kMaxProbs];
  int n, T, head;   // problems, tiles over all problems, index of the head problem (-1: none)
};

struct alignas(16) DfShared {
  DfPhase cph;                    // the consumers' current phase
  DfPhase pph;                    // the producer's current phase
  volatile int plan_layer;        // consumers started layer i: its weights may stream
  volatile int post_ready;        // the layer loop is over and the fields below are set
  volatile int abort;
  int post_hsm;                   // the HSM contractions run
  int n_ex;
  int fill_rows[DF_MAX_LAYERS + 1];   // rows of skipped-layer group r (tokens with i* < r)
  int flag;
  int scal[4];
  float best_v[3][kMaxB];          // per epilogue warp: best logit of each row so far
  int best_i[3][kMaxB];
  int xdst[kMaxB];
  float xw[kMaxB];
  float rs[3][DF_MAX_BATCH * 32];  // chunk partial sums of row reductions
  Epi epi_s[kStashProbs];          // this phase's epilogue descriptors (problems pi0 .. pi0 + n - 1)
  int stash_pi0, stash_np;
  alignas(16) float bias_s[kStashTiles][32];   // bias slices of the CTA's first tiles (16-byte copies)
  alignas(16) float resid_s[kStashResid][kMaxB][32];
  alignas(16) float2 rope_s[kRopeRows][64];    // (cos, sin) rows of the step's tokens
  int rowtok[kMaxB];               // active row -> token (sequence) of the current layer
  int extok[kMaxB];                // exit order -> token
  long long tbase[kMaxB];          // token's cache offset at layer 0 (-1: no block)
  float rtot[3][kMaxB];            // row totals of the last row reduction
#ifdef ADEPT_DF_TRACE
  long long pc[TB_N];
  long long wk[16];   // work time per phase kind (release of the previous barrier -> arrival)
  long long t_rel;
  int cur;
#endif
};

// ---------------------------------------------------------------------------- PTX
__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mb_init(uint64_t* b, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void mb_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mb_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
}
__device__ __forceinline__ bool mb_try(uint64_t* b, uint32_t par) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(su32(b)), "r"(par)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void tma3d(const CUtensorMap* tm, uint64_t* bar, void* dst, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::
          "r"(su32(dst)),
      "l"((uint64_t)tm), "r"(0), "r"(y), "r"(z), "r"(su32(bar))
      : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void cp_async8(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(su32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(su32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Barrier of the 224 consumer threads (the producer warp never joins it).
__device__ __forceinline__ void cons_sync() { asm volatile("bar.sync 1, 224;" ::: "memory"); }
__device__ __forceinline__ unsigned ld_vol(const unsigned* p) { return *(const volatile unsigned*)p; }
__device__ __forceinline__ int ld_vol(const int* p) { return *(const volatile int*)p; }

// Bounded wait on an mbarrier phase; false on time-out or abort.
__device__ bool mb_wait(uint64_t* bar, uint32_t par, DfShared& sh, unsigned* err) {
  if (mb_try(bar, par)) return true;
  const long long t0 = clock64();
  for (int n = 0;; ++n) {
    if (mb_try(bar, par)) return true;
    if (n > 8) __nanosleep(32);   // long waits back off (leave issue slots to working warps)
    if (sh.abort) return false;
    if (clock64() - t0 > kTimeout) {
      atomicOr(err, ERRW_TIMEOUT);
      sh.abort = 1;
      return false;
    }
  }
}

// Grid-wide barrier of the consumers (all CTAs are co-resident: cooperative launch).
// bar[0] counts arrivals over the whole step (barrier k completes at (k + 1) * grid);
// the CTA that merges the greedy tokens, last of all, sets it back to 0.  A CTA that
// sees the time-out bit (its own or another CTA's) leaves.
__device__ __forceinline__ unsigned ld_acq(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_rel(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ bool grid_sync(const DfPlan& P, unsigned& gen, DfShared& sh) {
  DF_CLK(t_sync);
#ifdef ADEPT_DF_TRACE
  if (threadIdx.x == 0) sh.wk[sh.cur] += t_sync - sh.t_rel;
#endif
  cons_sync();
  if (threadIdx.x == 0 && !sh.abort) {
    red_rel(&P.bar[0], 1u);
    const unsigned target = (gen + 1u) * gridDim.x;
    const long long t0 = clock64();
    while (ld_acq(&P.bar[0]) < target) {
      __nanosleep(20);
      if (ld_vol(P.err) & ERRW_TIMEOUT) {
        sh.abort = 1;
        break;
      }
      if (clock64() - t0 > kTimeout) {
        atomicOr(P.err, ERRW_TIMEOUT);
        sh.abort = 1;
        break;
      }
    }
  }
  cons_sync();
  DF_C(TB_SYNC, t_sync);
#ifdef ADEPT_DF_TRACE
  if (threadIdx.x == 0) {
    sh.pc[TB_NSYNC] += 1;
    sh.t_rel = clock64();
  }
#endif
  gen += 1u;
  return !sh.abort;
}

// ---------------------------------------------------------------------------- phases
__device__ void build_phase(DfPhase& f, const DfCall& c, int kind, int layer, const DfShared& sh, int rows) {
  const DfPlan& P = *c.P;
  f.n = 0;
  f.head = -1;
  auto add = [&](const CUtensorMap* map, const Epi* epi, int N, int K, int xblk, int r) {
    DfProb& p = f.p[f.n++];
    p.map = map;
    p.epi = epi;
    p.N = N;
    p.K = K;
    p.tiles = (N + kTN - 1) / kTN;
    p.S = (K + kSK - 1) / kSK;
    p.xblk = xblk;
    p.rows = r;
  };
  switch (kind) {
    case PH_QKV: add(&P.L[layer - 1].m_qkv, &P.L[layer - 1].e_qkv, P.nqkv, P.D, 0, rows); break;
    case PH_O: add(&P.L[layer - 1].m_o, &P.L[layer - 1].e_o, P.D, P.Dq, 0, rows); break;
    case PH_UP: add(&P.L[layer - 1].m_up, &P.L[layer - 1].e_up, P.up_rows, P.D, 0, rows); break;
    case PH_DOWN: add(&P.L[layer - 1].m_down, &P.L[layer - 1].e_down, P.D, P.F, 0, rows); break;
    case PH_H1: add(&P.m_h[0], &P.e_h[0], P.m1, P.D, 0, rows); break;
    case PH_H2: add(&P.m_h[1], &P.e_h[1], P.m2, P.m1, 0, rows); break;
    case PH_H3: add(&P.m_h[2], &P.e_h[2], P.m1, P.m2, 0, rows); break;
    case PH_H4: add(&P.m_h[3], &P.e_h[3], P.D, P.m1, 0, rows); break;
    default:
      for (int r = 3; r <= P.N; ++r)
        if (sh.fill_rows[r] > 0) add(&P.L[r - 1].m_kv, &P.L[r - 1].e_kv, 2 * P.Dkv, P.D, 0, sh.fill_rows[r]);
      f.head = f.n;
      add(&P.m_head, &P.e_head, P.V, P.D, 1, c.B);
      break;
  }
  int t = 0;
  for (int k = 0; k < f.n; ++k) {
    f.p[k].tile0 = t;
    t += f.p[k].tiles;
  }
  f.T = t;
}

// Whole tiles per CTA: CTA c takes tiles [c T / G, (c + 1) T / G) of the phase.
__device__ __forceinline__ int tile_start(int cta, int T, int G) { return cta * T / G; }   // cta * T < 2^31
// Problem holding phase tile t (problems are in tile order; pi only moves forward).
__device__ __forceinline__ int tile_problem(const DfPhase& f, int t, int pi) {
  while (t >= f.p[pi].tile0 + f.p[pi].tiles) ++pi;
  return pi;
}

// ---------------------------------------------------------------------------- producer
__device__ void producer(const DfCall& c, DfShared& sh, uint8_t* stages, uint64_t* full, uint64_t* empty) {
  const DfPlan& P = *c.P;

  int slot = 0;
  uint32_t ph = 0, issued = 0, last_par = 0;
  long long n_issued = 0;
  auto stream = [&](int kind, int layer) -> bool {
    DfPhase& f = sh.pph;
    build_phase(f, c, kind, layer, sh, 0);
    const int t0 = tile_start(blockIdx.x, f.T, gridDim.x), t1 = tile_start(blockIdx.x + 1, f.T, gridDim.x);
    int pi = 0;
    for (int t = t0; t < t1; ++t) {
      pi = tile_problem(f, t, pi);
      const DfProb& pr = f.p[pi];
      const int tl = t - pr.tile0;
      for (int s = 0; s < pr.S; ++s) {
        DF_CLK(t_e);
        if (n_issued >= c.ring && !mb_wait(&empty[slot], ph ^ 1u, sh, P.err)) return false;
        DF_P(TB_PEMPTY, t_e);
        ++n_issued;
        mb_expect(&full[slot], kStageBytes);
        tma3d(pr.map, &full[slot], stages + (size_t)slot * kStageBytes, tl * kTN, s * kKC);
        issued |= 1u << slot;
        last_par = (last_par & ~(1u << slot)) | (ph << slot);
        if (++slot == c.ring) {
          slot = 0;
          ph ^= 1u;
        }
      }
    }
    return true;
  };
  // bounded wait on a consumer-published flag
  auto wait_until = [&](auto cond) -> bool {
    const long long t0 = clock64();
#ifdef ADEPT_DF_TRACE
    struct Acc {
      DfShared& sh;
      long long t0;
      __device__ ~Acc() { sh.pc[TB_PFLAG] += clock64() - t0; }
    } acc_{sh, t0};
#endif
    while (!cond()) {
      __nanosleep(64);
      if (sh.abort) return false;
      if (clock64() - t0 > kTimeout) {
        atomicOr(P.err, ERRW_TIMEOUT);
        sh.abort = 1;
        return false;
      }
    }
    return true;
  };
  bool ok = true;
  for (int i = 1; i <= P.N && ok; ++i) {
    if (!wait_until([&] { return sh.plan_layer >= i || sh.post_ready; })) {
      ok = false;
      break;
    }
    if (sh.plan_layer < i) break;   // the loop ended before layer i
    ok = stream(PH_QKV, i) && stream(PH_O, i) && stream(PH_UP, i) && stream(PH_DOWN, i);
  }
  if (ok && wait_until([&] { return sh.post_ready != 0; })) {
    if (sh.post_hsm) ok = stream(PH_H1, 0) && stream(PH_H2, 0) && stream(PH_H3, 0) && stream(PH_H4, 0);
    if (ok) stream(PH_FILLHEAD, 0);
  }
  // every copy issued has landed before the CTA may exit
  for (int s = 0; s < c.ring; ++s) {
    if (!(issued >> s & 1u)) continue;
    const long long t0 = clock64();
    while (!mb_try(&full[s], (last_par >> s) & 1u)) {
      if (clock64() - t0 > kTimeout) {
        atomicOr(P.err, ERRW_TIMEOUT);
        break;
      }
    }
  }
}

// ---------------------------------------------------------------------------- row steps
// Rows are read in 128-float chunks: chunk g of R rows (row g / NC, NC = D / 128 chunks per
// row) belongs to consumer warp g % 7, one float4 per lane.  A row's sum is the warp sums
// of its chunks added in chunk order, so every CTA computes identical statistics.  The
// first pass reads through L1; the later passes over the same rows hit it.
constexpr int kChunk = 128;
constexpr int kCachedChunks = 8;   // chunks per warp held in registers by a row pass
constexpr int kMaxChunks = DF_MAX_BATCH * 32;   // chunk partials a row reduction can hold

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }

// a / d for 0 <= a, a + d < 2^22, with rcp = 1 / d: the quotient's fractional part is at
// least 0.5 / d away from an integer, above the float rounding of (a + 0.5) * rcp.
__device__ __forceinline__ int qdiv(int a, float rcp) { return __float2int_rz(((float)a + 0.5f) * rcp); }

// Butterfly sums of N values across the warp's lanes (N independent chains, interleaved).
template <int N>
__device__ __forceinline__ void warp_sum_n(float (&v)[N]) {
#pragma unroll
  for (int o = 16; o; o >>= 1)
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], o);
}

// Row totals of the chunk partials sh.rs[k][r * NC + c] (k < NV) into sh.rtot[k][r]: one
// warp per row, lanes over the chunks, butterfly sum.  All consumer threads call it.
template <int NV>
__device__ void rows_total_n(DfShared& sh, int R, int NC) {
  cons_sync();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int r = warp; r < R; r += kConsWarps) {
    float t[NV];
#pragma unroll
    for (int k = 0; k < NV; ++k) t[k] = 0.f;
    for (int cc = lane; cc < NC; cc += 32)
#pragma unroll
      for (int k = 0; k < NV; ++k) t[k] += sh.rs[k][r * NC + cc];
    warp_sum_n<NV>(t);
    if (lane == 0)
#pragma unroll
      for (int k = 0; k < NV; ++k) sh.rtot[k][r] = t[k];
  }
  cons_sync();
}

// Warp sums of per-lane chunk partials: p[i][k] is this lane's partial of value k for
// chunk g0 + warp + 7 i; the sums go to sh.rs[k][chunk] (chunks below g1 only).
template <int NV>
__device__ __forceinline__ void store_chunk_sums(DfShared& sh, float (&p)[kCachedChunks][NV], int g0, int g1) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 16; o; o >>= 1)
#pragma unroll
    for (int i = 0; i < kCachedChunks; ++i)
#pragma unroll
      for (int k = 0; k < NV; ++k) p[i][k] += __shfl_xor_sync(0xffffffffu, p[i][k], o);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kCachedChunks; ++i) {
      const int g = g0 + warp + kConsWarps * i;
      if (g < g1)
#pragma unroll
        for (int k = 0; k < NV; ++k) sh.rs[k][g] = p[i][k];
    }
  }
}

// This lane's float4 of each chunk g0 + warp + 7 i (zeros past g1).
__device__ __forceinline__ void load_chunks(const float* src, int D, int NC, int g0, int g1, float4 (&v)[kCachedChunks]) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float rnc = 1.f / NC;
#pragma unroll
  for (int i = 0; i < kCachedChunks; ++i) {
    const int g = g0 + warp + kConsWarps * i;
    if (g < g1) {
      const int r = qdiv(g, rnc), cc = g - r * NC;
      v[i] = ld4(src + (size_t)r * D + cc * kChunk + 4 * lane);
    } else {
      v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

constexpr int kBatchChunks = kConsWarps * kCachedChunks;

// Standardised rows (the family's attention-input normalisation; gains live in the
// weights) of an fp32 matrix into X as bf16, rows Kp apart.  Row sets of at most
// kBatchChunks chunks are read once and kept in registers; larger ones are read once per
// pass.  Mean, then the centred second moment (two passes, as the definition).
__device__ void std_rows(DfShared& sh, const float* src, int R, int D, int mode, float eps, bf16* X, int Kp) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int NC = D / kChunk, G = R * NC;
  const float rnc = 1.f / NC;
  const bool cached = G <= kBatchChunks;
  float4 v[kCachedChunks];
  DF_CLK(t_s0);
  if (cached) load_chunks(src, D, NC, 0, G, v);
#ifdef ADEPT_DF_TRACE
  if (cached) {
    float z = v[0].x + v[kCachedChunks - 1].x;
    asm volatile("" ::"f"(z));
  }
#endif
  DF_C(TB_SX_LOAD, t_s0);
  DF_CLK(t_s1);
  if (mode == NORM_LN) {
    for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
      if (!cached) load_chunks(src, D, NC, g0, G, v);
      float p[kCachedChunks][1];
#pragma unroll
      for (int i = 0; i < kCachedChunks; ++i) p[i][0] = (v[i].x + v[i].y) + (v[i].z + v[i].w);
      store_chunk_sums<1>(sh, p, g0, G);
    }
    rows_total_n<1>(sh, R, NC);
    if (threadIdx.x < (unsigned)R) sh.rtot[1][threadIdx.x] = sh.rtot[0][threadIdx.x] / D;   // means
  } else if (threadIdx.x < (unsigned)R) {
    sh.rtot[1][threadIdx.x] = 0.f;
  }
  DF_C(TB_SX_MEAN, t_s1);
  DF_CLK(t_s2);
  if (mode != NORM_COPY) {
    cons_sync();
    for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
      if (!cached) load_chunks(src, D, NC, g0, G, v);
      float p[kCachedChunks][1];
#pragma unroll
      for (int i = 0; i < kCachedChunks; ++i) {
        const int g = g0 + warp + kConsWarps * i;
        const float mu = g < G ? sh.rtot[1][qdiv(g, rnc)] : 0.f;
        const float a = v[i].x - mu, b = v[i].y - mu, c2 = v[i].z - mu, d = v[i].w - mu;
        p[i][0] = g < G ? (a * a + b * b) + (c2 * c2 + d * d) : 0.f;
      }
      store_chunk_sums<1>(sh, p, g0, G);
    }
    rows_total_n<1>(sh, R, NC);   // rtot[0] = centred sums of squares; rtot[1] = means
  }
  DF_C(TB_SX_VAR, t_s2);
  DF_CLK(t_s3);
  for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
    if (!cached) load_chunks(src, D, NC, g0, G, v);
#pragma unroll
    for (int i = 0; i < kCachedChunks; ++i) {
      const int g = g0 + warp + kConsWarps * i;
      if (g < G) {
        const int r = qdiv(g, rnc), cc = g - r * NC;
        float mu = 0.f, rstd = 1.f;
        if (mode != NORM_COPY) {
          mu = sh.rtot[1][r];
          rstd = rsqrtf(sh.rtot[0][r] / D + eps);
        }
        const __nv_bfloat162 lo = __floats2bfloat162_rn((v[i].x - mu) * rstd, (v[i].y - mu) * rstd);
        const __nv_bfloat162 hi = __floats2bfloat162_rn((v[i].z - mu) * rstd, (v[i].w - mu) * rstd);
        uint2 w;
        w.x = *reinterpret_cast<const uint32_t*>(&lo);
        w.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(X + (size_t)r * Kp + cc * kChunk + 4 * lane) = w;
      }
    }
  }
  DF_C(TB_SX_OUT, t_s3);
}

// bf16 rows into shared memory (16-byte pieces over every consumer thread).
__device__ void copy_rows(const bf16* src, int R, int K, int ld, bf16* X, int Kp) {
  const int n8 = K / 8;
  for (int r = 0; r < R; ++r) {
#pragma unroll 8
    for (int k = threadIdx.x; k < n8; k += kCons)
      *reinterpret_cast<uint4*>(X + (size_t)r * Kp + 8 * k) = *reinterpret_cast<const uint4*>(src + (size_t)r * ld + 8 * k);
  }
}

// HSM input (Sec. 4.2, Table S1): three separately RMS-normalised rows (shared gain g0)
// and the 3x3 convolution with padding (0, 1): c0[t] = b + sum_a sum_u w[a][u] x_a[t+u-1].
// c0 goes to shared memory (bf16, the FC1 operand) and, from CTA 0, to c0f (fp32).
__device__ void hsm_prep_rows(const DfPlan& P, DfShared& sh, int R, bf16* X, int Kp) {
  const int D = P.D, NC = D / kChunk, G = R * NC;
  const float* src[3] = {P.hsm_s, P.hsm_prev, P.hsm_I};
  for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
    float p[kCachedChunks][3];
#pragma unroll
    for (int a = 0; a < 3; ++a) {
      float4 v[kCachedChunks];
      load_chunks(src[a], D, NC, g0, G, v);
#pragma unroll
      for (int i = 0; i < kCachedChunks; ++i) p[i][a] = (v[i].x * v[i].x + v[i].y * v[i].y) + (v[i].z * v[i].z + v[i].w * v[i].w);
    }
    store_chunk_sums<3>(sh, p, g0, G);
  }
  rows_total_n<3>(sh, R, NC);
  const float* cv = P.hsm_conv;
  for (int r = 0; r < R; ++r)
  for (int t = threadIdx.x; t < D; t += kCons) {
    float acc = cv[9];
#pragma unroll
    for (int a = 0; a < 3; ++a) {
      const float* x = src[a] + (size_t)r * D;
      const float sc = rsqrtf(sh.rtot[a][r] / D + P.hsm_eps);
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int tt = t + u - 1;
        if (tt >= 0 && tt < D) acc += cv[a * 3 + u] * (x[tt] * sc * P.hsm_g0[tt]);
      }
    }
    X[(size_t)r * Kp + t] = __float2bfloat16_rn(acc);
    if (blockIdx.x == 0) P.c0f[(size_t)r * D + t] = acc;
  }
}

// h4 = RMSNorm_g1(h3) + h1 (the HSM MLP's addition), rounded for FC4.
__device__ void hsm_mid_rows(const DfPlan& P, DfShared& sh, int R, bf16* X, int Kp) {
  const int m1 = P.m1, NC = m1 / kChunk, G = R * NC;
  for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
    float4 v[kCachedChunks];
    load_chunks(P.h3f, m1, NC, g0, G, v);
    float p[kCachedChunks][1];
#pragma unroll
    for (int i = 0; i < kCachedChunks; ++i) p[i][0] = (v[i].x * v[i].x + v[i].y * v[i].y) + (v[i].z * v[i].z + v[i].w * v[i].w);
    store_chunk_sums<1>(sh, p, g0, G);
  }
  rows_total_n<1>(sh, R, NC);
  for (int r = 0; r < R; ++r)
  for (int d = threadIdx.x; d < m1; d += kCons) {
    const float sc = rsqrtf(sh.rtot[0][r] / m1 + P.hsm_eps);
    X[(size_t)r * Kp + d] =
        __float2bfloat16_rn(P.h3f[(size_t)r * m1 + d] * sc * P.hsm_g1[d] + P.h1f[(size_t)r * m1 + d]);
  }
}

// s~ = RMSNorm_g2(h5) + c0 (identity: s~ = s_i*) of exited row k -> the token's final
// state, and its standardised copy for the skipped-layer fills.  One CTA per row.
__device__ void hsm_out_row(const DfPlan& P, DfShared& sh, int k, int identity) {
  const int D = P.D, NC = D / kChunk;
  const int tok = sh.extok[k];
  float* f = P.final_ + (size_t)tok * D;
  const float* h5 = P.h5f + (size_t)k * D;
  float sc = 0.f;
  if (!identity) {
    for (int g0 = 0; g0 < NC; g0 += kBatchChunks) {
      float4 v[kCachedChunks];
      load_chunks(h5, D, NC, g0, NC, v);
      float p[kCachedChunks][1];
#pragma unroll
      for (int i = 0; i < kCachedChunks; ++i) p[i][0] = (v[i].x * v[i].x + v[i].y * v[i].y) + (v[i].z * v[i].z + v[i].w * v[i].w);
      store_chunk_sums<1>(sh, p, g0, NC);
    }
    rows_total_n<1>(sh, 1, NC);
    sc = rsqrtf(sh.rtot[0][0] / D + P.hsm_eps);
  }
  for (int d = threadIdx.x; d < D; d += kCons)
    f[d] = identity ? P.hsm_s[(size_t)k * D + d] : h5[d] * sc * P.hsm_g2[d] + P.c0f[(size_t)k * D + d];
  __threadfence_block();
  cons_sync();
  std_rows(sh, f, 1, D, P.norm_mode, P.eps, P.xfill + (size_t)k * D, D);
}

// Exit test (Sec. 4.1), stable compaction and row moves (App. I).  Every CTA computes
// the similarities and decisions of all active rows (identical arithmetic, so identical
// results); CTA 0 writes the bookkeeping; each CTA moves its slice of the columns.
__device__ void exit_phase(const DfCall& c, DfShared& sh, int layer, int par, int n, int& exited) {
  const DfPlan& P = *c.P;
  const int D = P.D, N = P.N, NC = D / kChunk, G = n * NC;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  const float* Xin = P.X_in[par];
  const float* Xout = P.X_out;
  const float* I = P.I[par];
  const int first = layer == 1, test = layer >= 2;
  // exits so far in this step: tracked by every CTA (CTA 0 rewrites the device counter
  // during this phase, so it is not read here)
  const int base = exited;
  const int* row_tok = sh.rowtok;
  for (int g0 = 0; g0 < G; g0 += kBatchChunks) {
    float4 va[kCachedChunks], vb[kCachedChunks];
    load_chunks(Xout, D, NC, g0, G, va);
    if (test) load_chunks(I, D, NC, g0, G, vb);
    float p[kCachedChunks][3];
#pragma unroll
    for (int i = 0; i < kCachedChunks; ++i) {
      const float4 a = va[i];
      p[i][0] = (a.x * a.x + a.y * a.y) + (a.z * a.z + a.w * a.w);
      if (test) {
        const float4 b = vb[i];
        p[i][1] = (b.x * b.x + b.y * b.y) + (b.z * b.z + b.w * b.w);
        p[i][2] = (a.x * b.x + a.y * b.y) + (a.z * b.z + a.w * b.w);
      } else {
        p[i][1] = p[i][2] = 0.f;
      }
    }
    store_chunk_sums<3>(sh, p, g0, G);
  }
  rows_total_n<3>(sh, n, NC);
  if (tid < n) {
    const int r = tid;
    const float ns = sh.rtot[0][r], ni = sh.rtot[1][r], dt = sh.rtot[2][r];
    const int tok = row_tok[r];
    int ex = 0;
    if (test) {
      const float cs = (ns > 0.f && ni > 0.f) ? dt / sqrtf(ns * ni) : -INFINITY;
      const int f = c.forced ? c.forced[tok] : 0;
      if (blockIdx.x == 0) {
        if (c.sim_out) c.sim_out[(size_t)tok * N + (layer - 1)] = cs;
        if (f != 0 && (f < 2 || f > N)) atomicOr(P.err, ERRW_FORCED);
      }
      ex = (f > 0) ? (f == layer) : (cs >= c.delta);
    }
    sh.xdst[r] = ex;
    sh.xw[r] = ns > 0.f ? rsqrtf(ns) : 0.f;
  }
  cons_sync();
  if (tid == 0) {
    int e = 0, k = 0;
    for (int r = 0; r < n; ++r) {
      const int tok = row_tok[r];
      if (sh.xdst[r]) {
        sh.xdst[r] = -1 - (base + e);
        sh.extok[base + e] = tok;
        if (blockIdx.x == 0) {
          P.exit_tok[base + e] = tok;
          if (c.exit_out) c.exit_out[tok] = layer;
        }
        ++e;
      } else {
        sh.xdst[r] = k;
        sh.rowtok[k] = tok;   // k <= r: entries not yet read are never overwritten
        if (blockIdx.x == 0) P.row_tok[par ^ 1][k] = tok;
        ++k;
      }
    }
    if (blockIdx.x == 0) {
      P.ctr[CTR_ACTIVE + (par ^ 1)] = k;
      P.ctr[CTR_EXITED] = base + e;
      P.ctr[CTR_PREFIX + layer] = base + e;
    }
    sh.scal[3] = base + e;
  }
  cons_sync();
  exited = sh.scal[3];
  // this CTA's columns (float4 units) of every row
  const int q4 = D / 4, cw = (q4 + gridDim.x - 1) / gridDim.x, q0 = blockIdx.x * cw;
  for (int r = 0; r < n; ++r)
  for (int q = q0 + tid; q < min(q4, q0 + cw); q += kCons) {
    const int d0 = sh.xdst[r];
    const float4 v = ld4(Xout + (size_t)r * D + 4 * q);
    const float4 in = ld4(I + (size_t)r * D + 4 * q);
    if (d0 >= 0) {
      const float w = sh.xw[r];
      float4 ni;
      ni.x = (first ? 0.f : in.x) + v.x * w;
      ni.y = (first ? 0.f : in.y) + v.y * w;
      ni.z = (first ? 0.f : in.z) + v.z * w;
      ni.w = (first ? 0.f : in.w) + v.w * w;
      *reinterpret_cast<float4*>(P.X_in[par ^ 1] + (size_t)d0 * D + 4 * q) = v;
      *reinterpret_cast<float4*>(P.I[par ^ 1] + (size_t)d0 * D + 4 * q) = ni;
    } else {
      const size_t kk = (size_t)(-1 - d0);
      *reinterpret_cast<float4*>(P.hsm_s + kk * D + 4 * q) = v;
      *reinterpret_cast<float4*>(P.hsm_prev + kk * D + 4 * q) = ld4(Xin + (size_t)r * D + 4 * q);
      *reinterpret_cast<float4*>(P.hsm_I + kk * D + 4 * q) = in;
    }
  }
}

// After layer N the remaining rows' s_N are their final states (column slices per CTA).
__device__ void final_phase(const DfCall& c, const DfShared& sh, int n) {
  const DfPlan& P = *c.P;
  const int D = P.D, q4 = D / 4, cw = (q4 + gridDim.x - 1) / gridDim.x, q0 = blockIdx.x * cw;
  for (int r = 0; r < n; ++r)
  for (int q = q0 + (int)threadIdx.x; q < min(q4, q0 + cw); q += kCons) {
    const int tok = sh.rowtok[r];
    *reinterpret_cast<float4*>(P.final_ + (size_t)tok * D + 4 * q) = ld4(P.X_out + (size_t)r * D + 4 * q);
  }
  if (blockIdx.x == 0 && (int)threadIdx.x < n && c.exit_out) c.exit_out[sh.rowtok[threadIdx.x]] = P.N;
}

// ---------------------------------------------------------------------------- attention
// One query row per sequence over the paged cache of one layer, split over the keys:
// warp item (row, head, split) covers `chunk` keys.  In a warp 8 keys are in flight per
// step, 4 lanes per key each owning a quarter of the head dimensions; the K and V rows of
// SUB steps are loaded before any is used.  The last split of a (row, head) to finish
// merges the partials in split order.
template <int DH>
__device__ void attention_phase(const DfCall& c, const DfShared& sh, int layer0, int n_act) {
  const DfPlan& P = *c.P;
  constexpr int PD = DH / 4;              // dimensions per lane
  constexpr int NV = PD / 8;              // 16-byte pieces per lane per row
  constexpr int SUB = DH == 64 ? 4 : 2;   // 8-key steps loaded together
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gk = lane >> 2, jq = lane & 3;
  const int H = P.H, nsplit = c.attn_nsplit, chunk = c.attn_chunk;
  const int group = H / P.Hkv;
  const int n_items = n_act * H * nsplit;
  const float scale = 1.4426950408889634f / sqrtf((float)DH);
  const bf16* Kp = (const bf16*)P.cache.k;
  const bf16* Vp = (const bf16*)P.cache.v;
  for (int it = blockIdx.x * kConsWarps + warp; it < n_items; it += gridDim.x * kConsWarps) {
    const int rh = it / nsplit, split = it - rh * nsplit;
    const int r = rh / H, h = rh - r * H;
    const int tok = sh.rowtok[r];
    const int sq = tok, pos = c.pos[tok];   // a generation step's token r is sequence r
    const int k_lo = split * chunk, k_hi = min(pos + 1, k_lo + chunk);
    const int kvh = h / group;
    float qv[PD];
    {
      const uint4* qp = reinterpret_cast<const uint4*>(P.q + (size_t)r * P.Dq + h * DH + jq * PD);
#pragma unroll
      for (int v = 0; v < NV; ++v) {
        const uint4 w = qp[v];
        const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&w);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(b2[e]);
          qv[8 * v + 2 * e] = f.x * scale;
          qv[8 * v + 2 * e + 1] = f.y * scale;
        }
      }
    }
    float m = -INFINITY, l = 0.f, o[PD];
#pragma unroll
    for (int d = 0; d < PD; ++d) o[d] = 0.f;
    for (int kb = k_lo; kb < k_hi; kb += 8 * SUB) {
      uint4 kr[SUB][NV], vr[SUB][NV];
      bool val[SUB];
#pragma unroll
      for (int u = 0; u < SUB; ++u) {
        const int key = kb + 8 * u + gk;
        val[u] = key < k_hi;
        if (val[u] && !DF_CHECK(P, P.cache.offset(layer0, sq, key, kvh) + DH <= (size_t)P.pool_elems, 3, key))
          val[u] = false;
        if (val[u]) {
          size_t off;
          if (P.bt_shift >= 0) {
            const KVCacheView& cv = P.cache;
            const int blk = cv.block_table[sq * cv.max_blocks_per_seq + (key >> P.bt_shift)];
            off = ((((size_t)layer0 * cv.n_blocks + blk) * cv.n_kv_heads + kvh) * cv.block_tokens +
                   (key & (cv.block_tokens - 1))) * (size_t)DH + jq * PD;
          } else {
            off = P.cache.offset(layer0, sq, key, kvh) + jq * PD;
          }
#pragma unroll
          for (int v = 0; v < NV; ++v) {
            kr[u][v] = *reinterpret_cast<const uint4*>(Kp + off + 8 * v);
            vr[u][v] = *reinterpret_cast<const uint4*>(Vp + off + 8 * v);
          }
        } else {
#pragma unroll
          for (int v = 0; v < NV; ++v) kr[u][v] = vr[u][v] = make_uint4(0, 0, 0, 0);
        }
      }
      float s[SUB];
      float mx = -INFINITY;
#pragma unroll
      for (int u = 0; u < SUB; ++u) {
        float a = 0.f;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&kr[u][v]);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(b2[e]);
            a = fmaf(qv[8 * v + 2 * e], f.x, a);
            a = fmaf(qv[8 * v + 2 * e + 1], f.y, a);
          }
        }
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        s[u] = val[u] ? a : -INFINITY;
        mx = fmaxf(mx, s[u]);
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      const float mn = fmaxf(m, mx);
      const float corr = (m == -INFINITY) ? 0.f : exp2f(m - mn);
      float p[SUB], ps = 0.f;
#pragma unroll
      for (int u = 0; u < SUB; ++u) {
        p[u] = val[u] ? exp2f(s[u] - mn) : 0.f;
        ps += p[u];
      }
      ps += __shfl_xor_sync(0xffffffffu, ps, 4);
      ps += __shfl_xor_sync(0xffffffffu, ps, 8);
      ps += __shfl_xor_sync(0xffffffffu, ps, 16);
      l = l * corr + ps;
#pragma unroll
      for (int d = 0; d < PD; ++d) o[d] *= corr;
#pragma unroll
      for (int u = 0; u < SUB; ++u) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&vr[u][v]);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(b2[e]);
            o[8 * v + 2 * e] = fmaf(p[u], f.x, o[8 * v + 2 * e]);
            o[8 * v + 2 * e + 1] = fmaf(p[u], f.y, o[8 * v + 2 * e + 1]);
          }
        }
      }
      m = mn;
    }
    // sum the 8 key groups of the warp
#pragma unroll
    for (int d = 0; d < PD; ++d) {
      o[d] += __shfl_xor_sync(0xffffffffu, o[d], 4);
      o[d] += __shfl_xor_sync(0xffffffffu, o[d], 8);
      o[d] += __shfl_xor_sync(0xffffffffu, o[d], 16);
    }
    float* w = P.attn_ws + ((size_t)rh * nsplit + split) * (DH + 2);
    if (gk == 0) {
#pragma unroll
      for (int d = 0; d < PD; ++d) w[jq * PD + d] = o[d];
    }
    if (lane == 0) {
      w[DH] = m;
      w[DH + 1] = l;
    }
    __threadfence();
    __syncwarp();
    unsigned last = 0;
    if (lane == 0) last = atomicAdd(P.attn_cnt + rh, 1u) == (unsigned)nsplit - 1u;
    last = __shfl_sync(0xffffffffu, last, 0);
    if (last) {
      __threadfence();
      const float* ws = P.attn_ws + (size_t)rh * nsplit * (DH + 2);
      float M = -INFINITY;
      for (int s2 = 0; s2 < nsplit; ++s2) M = fmaxf(M, __ldcg(ws + s2 * (DH + 2) + DH));
      float L = 0.f;
      for (int s2 = 0; s2 < nsplit; ++s2) {
        const float ms = __ldcg(ws + s2 * (DH + 2) + DH);
        if (ms != -INFINITY) L += exp2f(ms - M) * __ldcg(ws + s2 * (DH + 2) + DH + 1);
      }
      const float inv = L > 0.f ? 1.f / L : 0.f;
      constexpr int PL = DH / 32;
#pragma unroll
      for (int d = 0; d < PL; ++d) {
        float acc = 0.f;
        for (int s2 = 0; s2 < nsplit; ++s2) {
          const float ms = __ldcg(ws + s2 * (DH + 2) + DH);
          if (ms != -INFINITY) acc += exp2f(ms - M) * __ldcg(ws + s2 * (DH + 2) + lane * PL + d);
        }
        P.att[(size_t)r * P.Dq + h * DH + lane * PL + d] = __float2bfloat16_rn(acc * inv);
      }
      if (lane == 0) P.attn_cnt[rh] = 0u;
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------- contractions
// Operand X of a phase into shared memory: rows of Kp = K + 8 bf16 (the 16-byte pad
// spreads the rows of an n8 fragment over all banks).  Returns the element offset of the
// second operand block (the head rows of the fill + head phase).
__device__ int load_x(const DfCall& c, DfShared& sh, int kind, int par, int rows, bf16* X) {
  const DfPlan& P = *c.P;
  switch (kind) {
    case PH_QKV: std_rows(sh, P.X_in[par], rows, P.D, P.norm_mode, P.eps, X, P.D + 8); return 0;
    case PH_O: copy_rows(P.att, rows, P.Dq, P.Dq, X, P.Dq + 8); return 0;
    case PH_UP: std_rows(sh, P.X_out, rows, P.D, P.norm_mode, P.eps, X, P.D + 8); return 0;
    case PH_DOWN: copy_rows(P.hbuf, rows, P.F, P.F, X, P.F + 8); return 0;
    case PH_H1: hsm_prep_rows(P, sh, rows, X, P.D + 8); return 0;
    case PH_H2: copy_rows(P.h1t, rows, P.m1, P.m1, X, P.m1 + 8); return 0;
    case PH_H3: copy_rows(P.h2t, rows, P.m2, P.m2, X, P.m2 + 8); return 0;
    case PH_H4: hsm_mid_rows(P, sh, rows, X, P.m1 + 8); return 0;
    default: {
      const int ne = sh.n_ex;
      copy_rows(P.xfill, ne, P.D, P.D, X, P.D + 8);
      const int off1 = ne * (P.D + 8);
      std_rows(sh, P.final_, c.B, P.D, P.norm_mode, P.eps, X + off1, P.D + 8);
      return off1;
    }
  }
}

// Cache facts of GEMM row r for the KV-writing epilogues, from the step's per-token
// facts in shared memory (no dependent global loads): QKV rows are the active rows of the
// layer, KV (fill) rows are the exited tokens in exit order.
__device__ __forceinline__ EpiRow fast_row(const Epi& e, int r, const DfShared& sh, const DfCall& c) {
  EpiRow rr{-1, 0, nullptr};
  if (e.kind == EPI_QKV || e.kind == EPI_KV) {
    const int tok = e.kind == EPI_QKV ? sh.rowtok[r] : sh.extok[r];
    rr.pos = c.pos[tok];
    const long long b0 = sh.tbase[tok];
    rr.cbase = b0 < 0 ? -1 : b0 + (long long)e.layer0 * c.lstride;
    if (e.rope && tok < kRopeRows) rr.rope = sh.rope_s[tok];
  }
  return rr;
}

// Epilogue of one finished 32-column tile by one warp: res[j * rb + row] is column j of
// row; lane r handles row r.  it: the tile's index among the CTA's tiles of the phase
// (selects the staged bias / residual slices).
__device__ void tile_epilogue(const DfCall& c, const DfShared& sh, const DfProb& pr, int pi, int t, int it,
                              const float* res, int rb, float* best_v, int* best_i, bool head) {
  const int r = threadIdx.x & 31;
  if (r >= pr.rows) return;
  float v[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = res[j * rb + r];
  const int si = pi - sh.stash_pi0;
  const Epi& e = (si >= 0 && si < sh.stash_np) ? sh.epi_s[si] : *pr.epi;
  const EpiRow rr = fast_row(e, r, sh, c);
  if (e.kind == EPI_QKV || e.kind == EPI_KV) {
    const long long span = (long long)(e.n_kv_cols / e.head_dim - 1) * e.cache.head_stride() + e.head_dim;
    if (!DF_CHECK(*c.P, rr.cbase < 0 || rr.cbase + span <= c.P->pool_elems, 1, (unsigned)t)) return;
  }
  if (!DF_CHECK(*c.P, t * kTN < pr.N && r < kMaxB, 2, (unsigned)t)) return;
  const float* b32 = (e.bias && it < kStashTiles && t * kTN + kTN <= pr.N) ? sh.bias_s[it] : nullptr;
  const float* r32 = (e.kind == EPI_RESID && it < kStashResid) ? sh.resid_s[it][r] : nullptr;
  epi_chunk32<bf16>(e, r, t * kTN, pr.N, v, rr, b32, r32);
  if (head) {
    float bv = best_v[r];
    int bi = best_i[r];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int col = t * kTN + j;
      if (col < pr.N && (v[j] > bv || (v[j] == bv && col < bi))) {
        bv = v[j];
        bi = col;
      }
    }
    best_v[r] = bv;
    best_i[r] = bi;
  }
}

// Epilogue warps, at the start of a phase: copy the CTA's epilogue descriptors and the
// bias / residual slices of its first tiles into shared memory (asynchronous copies that
// overlap the operand staging; waited for before the phase's MMA loop starts).
__device__ void stage_epilogue(const DfCall& c, DfShared& sh, int t0, int t1) {
  const DfPhase& f = sh.cph;
  const int et = threadIdx.x - kMmaWarps * 32;   // 0..95
  if (t0 >= t1) return;
  const int pi0 = tile_problem(f, t0, 0), pi1 = tile_problem(f, t1 - 1, pi0);
  const int np = min(pi1 - pi0 + 1, kStashProbs);
  if (et == 0) {
    sh.stash_pi0 = pi0;
    sh.stash_np = np;
  }
  constexpr int E8 = (int)(sizeof(Epi) / 8);
  for (int i = et; i < np * E8; i += 96) {
    const int k = i / E8, w = i - k * E8;
    cp_async8(reinterpret_cast<uint64_t*>(&sh.epi_s[k]) + w, reinterpret_cast<const uint64_t*>(f.p[pi0 + k].epi) + w);
  }
  // bias and residual slices (descriptor fields read from global once)
  const int nt = min(t1 - t0, kStashTiles);
  int pi = pi0;
  for (int i = 0; i < nt; ++i) {
    const int t = t0 + i;
    pi = tile_problem(f, t, pi);
    const DfProb& pr = f.p[pi];
    const Epi* e = pr.epi;
    const int c0 = (t - pr.tile0) * kTN;
    const float* bias = e->bias;
    // whole 32-column slices only (the last tile of a ragged width reads its bias in place)
    if (bias && c0 + kTN <= pr.N && et < 8) cp_async16(&sh.bias_s[i][4 * et], bias + c0 + 4 * et);
    if (i < kStashResid && e->kind == EPI_RESID) {
      const float* rs = e->resid;
      const int ld = e->ld_resid;
      for (int j = et; j < pr.rows * 8; j += 96) {
        const int r = j >> 3, q = j & 7;
        cp_async16(&sh.resid_s[i][r][4 * q], rs + (size_t)r * ld + c0 + 4 * q);
      }
    }
  }
}

// One contraction phase on the consumer side; the CTA owns whole tiles.  Warps 0..3
// (MMA): a tile's stages are dealt round-robin (stage k to warp k % 4), each consumed
// whole -- per 64-k chunk all fragments are loaded first, then the MMAs of two
// accumulator chains -- and the partial sums go to reduction buffer (tile # % 3).
// Warps 4..6 (epilogue): buffer b belongs to warp 4 + b, which sums the four partials,
// frees the buffer and runs the fused epilogue while the MMA warps go on.
__device__ bool gemm_phase(const DfCall& c, DfShared& sh, int kind, int layer, int par, int rows, uint8_t* stages,
                           uint64_t* full, uint64_t* empty, uint64_t* ready, uint64_t* freeb, bf16* X, float* red,
                           float* res, unsigned& cpos, unsigned& qseg) {
  const DfPlan& P = *c.P;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = c.rb;
  DF_CLK(t_lx);
  if (tid == 0) build_phase(sh.cph, c, kind, layer, sh, rows);
  if (kind == PH_FILLHEAD && tid < 3 * kMaxB) {
    sh.best_v[tid / kMaxB][tid % kMaxB] = -INFINITY;
    sh.best_i[tid / kMaxB][tid % kMaxB] = 0x7fffffff;
  }
  const int off1 = load_x(c, sh, kind, par, rows, X);
  cons_sync();
  DF_C(TB_LOADX, t_lx);
  const DfPhase& f = sh.cph;
  const int G = gridDim.x, cta = blockIdx.x;
  const int t0 = tile_start(cta, f.T, G), t1 = tile_start(cta + 1, f.T, G);
  if (warp >= kMmaWarps) {
    // the epilogue warps stage their operands while the MMA warps start the first tile
    stage_epilogue(c, sh, t0, t1);
    cp_async_wait_all();
    asm volatile("bar.sync 2, 96;" ::: "memory");
  }
  if (warp < kMmaWarps) {
    // this warp's ring position: stage k of the tile at slot (pos + k) mod ring
    int wslot = (int)(cpos % (unsigned)c.ring);   // once per phase
    uint32_t wph = (cpos / (unsigned)c.ring) & 1u;
    unsigned q = qseg;
    const int g4 = lane >> 2, tq = lane & 3;
    int pi = 0;
    for (int t = t0; t < t1; ++t, ++q) {
      DF_CLK(t_mma);
      pi = tile_problem(f, t, pi);
      const DfProb& pr = f.p[pi];
      const unsigned b = q % 3, use = q / 3;
      if (use > 0) {
        DF_CLK(t_fr);
        bool got = true;
        if (lane == 0) got = mb_wait(&freeb[b], (use - 1) & 1u, sh, P.err);
        DF_C(TB_FREEWAIT, t_fr);
        if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) break;
      }
      float acc[2][2][2][4];
#pragma unroll
      for (int a0 = 0; a0 < 2; ++a0)
#pragma unroll
        for (int a1 = 0; a1 < 2; ++a1)
#pragma unroll
          for (int a2 = 0; a2 < 2; ++a2)
#pragma unroll
            for (int a3 = 0; a3 < 4; ++a3) acc[a0][a1][a2][a3] = 0.f;
      const bf16* xs = X + (pr.xblk ? off1 : 0);
      const int Kp = pr.K + 8;
      const int nrow = pr.rows;
      const int K = pr.K;
      bool ok = true;
      // position of stage `warp` of this tile; later stages advance by 4 slots
      int slot = wslot + warp;
      uint32_t ph = wph;
      while (slot >= c.ring) {
        slot -= c.ring;
        ph ^= 1u;
      }
      for (int k = warp; k < pr.S; k += kMmaWarps) {
        DF_CLK(t_fw);
        bool got = true;
        if (lane == 0) got = mb_wait(&full[slot], ph, sh, P.err);
        ok = __shfl_sync(0xffffffffu, got ? 1 : 0, 0) != 0;
        DF_C(TB_FULLWAIT, t_fw);
        if (!ok) break;
        const uint32_t sb = su32(stages + (size_t)slot * kStageBytes);
#pragma unroll
        for (int ch = 0; ch < kKC; ++ch) {
          const int kb = k * kSK + ch * 64;
          if (kb >= K) break;
          const uint32_t cb = sb + ch * (kTN * 128);
#pragma unroll
          for (int kp = 0; kp < 4; kp += 2) {
            uint32_t a[2][2][4];
            uint32_t bf[2][2][2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int kk = kp + h;
#pragma unroll
              for (int mt = 0; mt < 2; ++mt) {
                const int mi = lane >> 3;
                const int row = mt * 16 + (lane & 7) + ((mi & 1) << 3);
                const int unit = kk * 2 + (mi >> 1);
                ldsm_x4(a[h][mt], cb + row * 128 + ((unit ^ (row & 7)) << 4));
              }
#pragma unroll
              for (int gr = 0; gr < 2; ++gr) {
                const int tok = gr * 8 + g4;
                bf[h][gr][0] = bf[h][gr][1] = 0u;
                if (tok < nrow) {
                  const uint32_t* xr =
                      reinterpret_cast<const uint32_t*>(xs + (size_t)tok * Kp + kb + kk * 16 + 2 * tq);
                  bf[h][gr][0] = xr[0];
                  bf[h][gr][1] = xr[4];
                }
              }
            }
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
              for (int gr = 0; gr < 2; ++gr) {
                if (gr * 8 >= nrow) break;
#pragma unroll
                for (int mt = 0; mt < 2; ++mt) mma16816(acc[h][mt][gr], a[h][mt], bf[h][gr][0], bf[h][gr][1]);
              }
          }
        }
        __syncwarp();
        if (lane == 0) mb_arrive(&empty[slot]);
        slot += kMmaWarps;
        while (slot >= c.ring) {
          slot -= c.ring;
          ph ^= 1u;
        }
      }
      // this warp's partial sums -> red[b][warp][n][tok]
      float* rw = red + ((size_t)(b * kMmaWarps + warp) * kTN) * rb;
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int gr = 0; gr < 2; ++gr) {
          if (gr * 8 >= rb) break;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int n = mt * 16 + g4 + ((k & 2) ? 8 : 0);
            const int tok = gr * 8 + 2 * tq + (k & 1);
            rw[n * rb + tok] = acc[0][mt][gr][k] + acc[1][mt][gr][k];
          }
        }
      __syncwarp();
      if (lane == 0) mb_arrive(&ready[b]);
      wslot += pr.S;   // the tile's stages
      while (wslot >= c.ring) {
        wslot -= c.ring;
        wph ^= 1u;
      }
      DF_C(TB_MMA, t_mma);
      if (!ok) break;
    }
  } else {
    const int e = warp - kMmaWarps;   // 0..2: owns buffer e
    float* rs = res + (size_t)e * kTN * rb;
    unsigned q = qseg;
    int pi = 0;
    for (int t = t0; t < t1; ++t, ++q) {
      const unsigned b = q % 3, use = q / 3;
      if ((int)b != e) continue;
      pi = tile_problem(f, t, pi);
      const DfProb& pr = f.p[pi];
      DF_CLK(t_rw);
      bool got = true;
      if (lane == 0) got = mb_wait(&ready[b], use & 1u, sh, P.err);
      DF_E(TB_REDUCE, t_rw);
      if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) break;
      DF_CLK(t_epi);
      const float* rd = red + ((size_t)b * kMmaWarps * kTN) * rb;
      for (int i = lane; i < kTN * rb; i += 32) {
        float a = 0.f;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w) a += rd[(size_t)w * kTN * rb + i];
        rs[i] = a;
      }
      __syncwarp();
      if (lane == 0) mb_arrive(&freeb[b]);
      tile_epilogue(c, sh, pr, pi, t - pr.tile0, t - t0, rs, rb, sh.best_v[e], sh.best_i[e], pi == f.head);
      __syncwarp();
      DF_E(TB_EPI, t_epi);
#ifdef ADEPT_DF_TRACE
      if (threadIdx.x == 128) sh.pc[TB_NFULL] += 1;
#endif
    }
  }
  // every consumer thread advances the same counters
  {
    int pi = 0;
    unsigned st = 0;
    for (int t = t0; t < t1; ++t) {
      pi = tile_problem(f, t, pi);
      st += f.p[pi].S;
    }
    cpos += st;
    qseg += (unsigned)(t1 - t0);
  }
  cons_sync();
  return !sh.abort;
}

// ---------------------------------------------------------------------------- consumers
__device__ void consumers(const DfCall& c, DfShared& sh, uint8_t* stages, uint64_t* full, uint64_t* empty,
                          uint64_t* ready, uint64_t* freeb, bf16* X, float* red, float* res) {
  const DfPlan& P = *c.P;
  const int tid = threadIdx.x;
  const int G = gridDim.x, cta = blockIdx.x;
  const int N = P.N, D = P.D, B = c.B;
  unsigned gen = 0;   // barriers passed in this step
  unsigned cpos = 0;   // stages consumed in this step
  unsigned qseg = 0;
  // layer 1 always runs (B >= 1): its weights may stream while the embeddings are set up
  if (tid == 0) sh.plan_layer = 1;
  DF_CLK(t_total);
  DF_CLK(t_emb);

  // ---- step set-up: counters, positions, embeddings s_0 (one CTA per sequence)
  if (cta == 0) {
    for (int e = tid; e < ctr_words(N); e += kCons) P.ctr[e] = e == CTR_ACTIVE ? B : 0;
    for (int e = tid; e < kMaxB * P.H; e += kCons) P.attn_cnt[e] = 0u;
    if (tid == 0) *P.amax_cnt = 0u;
  }
  // per-token facts every CTA keeps for the step: row map, exit order, cache base
  if (tid < B) {
    sh.rowtok[tid] = tid;
    sh.extok[tid] = 0;
    sh.tbase[tid] = P.cache.checked_base(0, tid, c.pos[tid]);
  }
  if (P.rope_table) {
    const int half = P.dh / 2;
    for (int e = tid; e < min(B, kRopeRows) * half; e += kCons) {
      const int b = e / half, j = e - b * half;
      sh.rope_s[b][j] = P.rope_table[(size_t)c.pos[b] * half + j];
    }
  }
  if (cta < B) {
    const int r = cta;
    if (tid == 0) {
      int p = c.pos[r];
      P.seq_len[r] = p + 1;
      if (p >= P.seq_cap || (P.max_pos > 0 && p >= P.max_pos)) {
        atomicOr(P.err, ERRW_POS);
        p = 0;
      }
      P.tok_seq[r] = r;
      P.tok_pos[r] = p;
      P.row_tok[0][r] = r;
      int tok = c.tokens[r];
      if (tok < 0 || tok >= P.V) {
        atomicOr(P.err, ERRW_TOKEN);
        tok = 0;
      }
      sh.scal[0] = p;
      sh.scal[1] = tok;
    }
    cons_sync();
    const int p = sh.scal[0], tok = sh.scal[1];
    float* x = P.X_in[0] + (size_t)r * D;
    for (int d = tid; d < D; d += kCons) {
      float v = __bfloat162float(P.tok_emb[(size_t)tok * D + d]);
      if (P.pos_emb) v += __bfloat162float(P.pos_emb[(size_t)p * D + d]);
      x[d] = v;
    }
    if (c.sim_out)
      for (int l = tid; l < N; l += kCons) c.sim_out[(size_t)r * N + l] = __int_as_float(0x7fffffff);
  }
  DF_C(TB_EMBED, t_emb);
  if (!grid_sync(P, gen, sh)) return;

  // ---- the layers
  int par = 0, i_end = N + 1, exited = 0;
  for (int i = 1; i <= N; ++i) {
    const int n_act = min(ld_vol(P.ctr + CTR_ACTIVE + par), kMaxB);
    if (n_act <= 0) {
      i_end = i;
      break;
    }
    if (tid == 0) sh.plan_layer = i;
    DF_PH(WK_QKV);
    if (!gemm_phase(c, sh, PH_QKV, i, par, n_act, stages, full, empty, ready, freeb, X, red, res, cpos, qseg))
      return;
    if (!grid_sync(P, gen, sh)) return;
    DF_PH(WK_ATTN);
    DF_CLK(t_at);
    if (P.dh == 64) attention_phase<64>(c, sh, i - 1, n_act);
    else attention_phase<128>(c, sh, i - 1, n_act);
    DF_C(TB_ATTN, t_at);
    if (!grid_sync(P, gen, sh)) return;
    DF_PH(WK_O);
    if (!gemm_phase(c, sh, PH_O, i, par, n_act, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
    if (!grid_sync(P, gen, sh)) return;
    DF_PH(WK_UP);
    if (!gemm_phase(c, sh, PH_UP, i, par, n_act, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
    if (!grid_sync(P, gen, sh)) return;
    DF_PH(WK_DOWN);
    if (!gemm_phase(c, sh, PH_DOWN, i, par, n_act, stages, full, empty, ready, freeb, X, red, res, cpos, qseg))
      return;
    if (!grid_sync(P, gen, sh)) return;
    DF_PH(i < N ? WK_EXIT : WK_FINAL);
    DF_CLK(t_ex);
    if (i < N) exit_phase(c, sh, i, par, n_act, exited);
    else final_phase(c, sh, n_act);
    DF_C(TB_EXIT, t_ex);
    if (!grid_sync(P, gen, sh)) return;
    if (i < N) par ^= 1;
  }

  // ---- after the loop: the HSM of the exited tokens, their fills, the head
  const int n_ex = min(ld_vol(P.ctr + CTR_EXITED), kMaxB);
  if (tid == 0) {
    sh.n_ex = n_ex;
    sh.post_hsm = n_ex > 0 && !c.identity;
    for (int r = 0; r <= N; ++r) {
      int rows = 0;
      if (r >= 3) {
        const int j = r - 1;   // tokens with i* <= j, i.e. i* < r
        rows = j < i_end ? ld_vol(P.ctr + CTR_PREFIX + j) : n_ex;
      }
      sh.fill_rows[r] = min(rows, n_ex);
    }
    __threadfence_block();
    sh.post_ready = 1;
  }
  cons_sync();
  if (n_ex > 0) {
    if (!c.identity) {
      DF_PH(WK_H1);
      if (!gemm_phase(c, sh, PH_H1, 0, 0, n_ex, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
      if (!grid_sync(P, gen, sh)) return;
      DF_PH(WK_H2);
      if (!gemm_phase(c, sh, PH_H2, 0, 0, n_ex, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
      if (!grid_sync(P, gen, sh)) return;
      DF_PH(WK_H3);
      if (!gemm_phase(c, sh, PH_H3, 0, 0, n_ex, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
      if (!grid_sync(P, gen, sh)) return;
      DF_PH(WK_H4);
      if (!gemm_phase(c, sh, PH_H4, 0, 0, n_ex, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;
      if (!grid_sync(P, gen, sh)) return;
    }
    DF_PH(WK_OUT);
    DF_CLK(t_ho);
    if (cta < n_ex) hsm_out_row(P, sh, cta, c.identity);
    DF_C(TB_HSMOUT, t_ho);
    if (!grid_sync(P, gen, sh)) return;
  }
  DF_PH(WK_FILLHEAD);
  if (!gemm_phase(c, sh, PH_FILLHEAD, 0, 0, B, stages, full, empty, ready, freeb, X, red, res, cpos, qseg)) return;

  // ---- greedy token: per-CTA best of each row, merged by the last CTA (lowest index on ties)
  DF_CLK(t_am);
  if (tid < B) {
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int e = 0; e < 3; ++e) {
      const float v = sh.best_v[e][tid];
      const int ix = sh.best_i[e][tid];
      if (v > bv || (v == bv && ix < bi)) {
        bv = v;
        bi = ix;
      }
    }
    P.amax_v[cta * kMaxB + tid] = bv;
    P.amax_i[cta * kMaxB + tid] = bi;
  }
  __threadfence();
  cons_sync();
  if (tid == 0) sh.flag = atomicAdd(P.amax_cnt, 1u) == (unsigned)G - 1u;
  cons_sync();
  if (sh.flag) {
    __threadfence();
    if (tid < B) {
      float bv = -INFINITY;
      int bi = 0x7fffffff;
      for (int k = 0; k < G; ++k) {
        const float v = __ldcg(P.amax_v + k * kMaxB + tid);
        const int ix = __ldcg(P.amax_i + k * kMaxB + tid);
        if (v > bv || (v == bv && ix < bi)) {
          bv = v;
          bi = ix;
        }
      }
      c.next_out[tid] = bi == 0x7fffffff ? 0 : bi;
    }
    if (tid == 0) {
      *P.amax_cnt = 0u;
      *(volatile unsigned*)P.bar = 0u;   // every CTA has passed every barrier of the step
    }
  }
  DF_C(TB_ARGMAX, t_am);
  DF_C(TB_TOTAL, t_total);
#ifdef ADEPT_DF_TRACE
  if (tid == 0) sh.wk[WK_FILLHEAD] += clock64() - sh.t_rel;
#endif
}

__global__ void __launch_bounds__(kThreads, 1) df_kernel(const __grid_constant__ DfCall c) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ DfShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* stages = base;
  bf16* X = reinterpret_cast<bf16*>(base + (size_t)c.ring * kStageBytes);
  float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(X) + c.x_bytes);
  float* res = red + 3 * kMmaWarps * kTN * c.rb;
  uint64_t* full = reinterpret_cast<uint64_t*>(res + 3 * kTN * c.rb);
  uint64_t* empty = full + c.ring;
  uint64_t* ready = empty + c.ring;
  uint64_t* freeb = ready + 3;
  const DfPlan& P = *c.P;
  if (threadIdx.x == 0) {
    for (int s = 0; s < c.ring; ++s) {
      mb_init(&full[s], 1);
      mb_init(&empty[s], 1);
    }
    for (int b = 0; b < 3; ++b) {
      mb_init(&ready[b], kMmaWarps);
      mb_init(&freeb[b], 1);
    }
    sh.plan_layer = 0;
    sh.post_ready = 0;
#ifdef ADEPT_DF_TRACE
    for (int k = 0; k < TB_N; ++k) sh.pc[k] = 0;
    for (int k = 0; k < 16; ++k) sh.wk[k] = 0;
    sh.cur = WK_EMBED;
    sh.t_rel = clock64();
#endif
    sh.abort = (ld_vol(P.err) & ERRW_TIMEOUT) ? 1 : 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (sh.abort) return;
  if (threadIdx.x >= kCons) {
    if (threadIdx.x == kCons) producer(c, sh, stages, full, empty);
#ifdef ADEPT_DF_TRACE
    __syncwarp();   // the producer lane rejoins its warp before the block-wide barrier below
#endif
  } else {
    consumers(c, sh, stages, full, empty, ready, freeb, X, red, res);
  }
#ifdef ADEPT_DF_TRACE
  __syncthreads();
  const int slot = blockIdx.x == 0 ? 0 : (blockIdx.x == gridDim.x / 2 ? 1 : -1);
  if (slot >= 0 && threadIdx.x < TB_N) g_df_prof[slot][threadIdx.x] = (unsigned long long)sh.pc[threadIdx.x];
  if (blockIdx.x < 256 && threadIdx.x < 16) g_df_work[blockIdx.x][threadIdx.x] = (unsigned long long)sh.wk[threadIdx.x];
#endif
}

}  // namespace

// ---------------------------------------------------------------------------- host
#ifdef ADEPT_DF_TRACE
static unsigned* g_dbg_words = nullptr;   // debug builds: self-check words of the last plan
#endif
struct DfState {
  DfPlan* dplan = nullptr;
  DfLayerDev* dlayers = nullptr;
  std::vector<void*> allocs;
  int grid = 0, ring = 0, x_bytes = 0, smem = 0, b_max = 0, H = 0, max_batch = 0, rb = 8;
  long long lstride = 0;
};

// Device memory for plans (they hold the TMA tensor maps the kernel reads from global
// memory): taken from blocks that are never freed, so no plan's maps ever sit at an address
// that held an earlier plan's maps -- a map cached by the TMA unit for a freed plan can
// never be mistaken for a new one.  A model load takes tens of KB.
static std::mutex g_arena_mu;
static char* g_arena = nullptr;
static size_t g_arena_left = 0;
static int g_arena_dev = -1;
static void* arena_alloc(size_t bytes) {
  std::lock_guard<std::mutex> lock(g_arena_mu);
  int dev = 0;
  cudaGetDevice(&dev);
  bytes = (bytes + 255) & ~(size_t)255;
  if (dev != g_arena_dev || bytes > g_arena_left) {
    const size_t sz = std::max(bytes, (size_t)4 << 20);
    void* p = nullptr;
    if (cudaMalloc(&p, sz) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    g_arena = (char*)p;
    g_arena_left = sz;
    g_arena_dev = dev;
  }
  void* p = g_arena;
  g_arena += bytes;
  g_arena_left -= bytes;
  return p;
}

static bool dmalloc(DfState* d, void** p, size_t bytes) {
  if (cudaMalloc(p, bytes) != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return false;
  }
  d->allocs.push_back(*p);
  return cudaMemset(*p, 0, bytes) == cudaSuccess;
}

static Epi epi0() {
  Epi e;
  memset(&e, 0, sizeof e);
  return e;
}

void df_destroy(DfState* d) {
  if (!d) return;
  for (void* p : d->allocs) cudaFree(p);
  delete d;
}

DfState* df_create(const DfModelSrc& s, std::string* why) {
  auto no = [&](const char* m) -> DfState* {
    if (why) *why = m;
    return nullptr;
  };
  if (!tc_gemm_supported()) return no("no sm_100-family device or tensor-map encoder");
  if (s.family != ADEPT_FAMILY_LLAMA && s.family != ADEPT_FAMILY_GPT2) return no("decoder families only");
  if (s.N < 3 || s.N > DF_MAX_LAYERS) return no("layer count outside [3, 64]");
  if (s.dh != 64 && s.dh != 128) return no("head_dim must be 64 or 128");
  if (s.D % 128 || s.m1 % 128 || s.Dq % 64 || s.F % 64 || s.m2 % 64)
    return no("widths must be multiples of 64 (d_model and the HSM's first width of 128)");
  const int nqkv = s.Dq + 2 * s.Dkv;
  if (nqkv % 32 || (2 * s.Dkv) % 32 || s.L[0].up_rows % 32) return no("projection widths must be multiples of 32");
  int dev = 0, nsm = 0, coop = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
  if (!coop || nsm <= 0) return no("no cooperative launch");
  // shared memory: X rows + the stage ring + reduction buffers + barriers
  const int kmax = std::max({s.D, s.Dq, s.F, s.m1, s.m2});
  const int budget = 232448 - (int)sizeof(DfShared) - 512;
  int b_max = 0, ring = 0, xb = 0, rb = 8, fixed = 0;
  for (int b = std::min(kMaxB, s.max_batch); b >= 1; --b) {
    if (b * (std::max(s.D, s.m1) / kChunk) > kMaxChunks) continue;
    const int rbb = b <= 8 ? 8 : 16;
    const int fx = 3 * (kMmaWarps + 1) * kTN * rbb * 4 + 6 * 8 + 1024;
    const int x = std::max(b * (kmax + 8) * 2, 2 * b * (s.D + 8) * 2);
    const int left = budget - fx - x;
    const int r = std::min(16, left / (kStageBytes + 16));
    if (r >= 4) {
      b_max = b;
      ring = r;
      xb = (x + 15) & ~15;
      rb = rbb;
      fixed = fx;
      break;
    }
  }
  if (b_max == 0) return no("operand rows do not fit shared memory");
  DfState* d = new DfState();
  d->ring = ring;
  d->x_bytes = xb;
  d->b_max = b_max;
  d->rb = rb;
  d->H = s.H;
  d->max_batch = s.max_batch;
  d->smem = ring * kStageBytes + xb + fixed + 2 * ring * 8;
  if (cudaFuncSetAttribute(df_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, d->smem) != cudaSuccess) {
    cudaGetLastError();
    df_destroy(d);
    return no("shared-memory attribute refused");
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, df_kernel, kThreads, d->smem) != cudaSuccess ||
      per_sm < 1) {
    cudaGetLastError();
    df_destroy(d);
    return no("kernel does not fit an SM");
  }
  d->grid = nsm;

  DfPlan h;
  memset(&h, 0, sizeof h);
  std::vector<DfLayerDev> hl(s.N);
  memset(hl.data(), 0, sizeof(DfLayerDev) * s.N);
  const int D = s.D;
  bool ok = true;
  auto map = [&](CUtensorMap* m, const void* w, int rows, int K) {
    ok = ok && tc_encode_weight_3d(m, w, K, rows, (size_t)K * 2, kTN, kKC);
  };
  for (int l = 0; l < s.N; ++l) {
    const DfLayerSrc& w = s.L[l];
    DfLayerDev& L = hl[l];
    const int par = l & 1;
    map(&L.m_qkv, w.w_qkv, nqkv, D);
    map(&L.m_o, w.w_o, D, s.Dq);
    map(&L.m_up, w.w_up, w.up_rows, D);
    map(&L.m_down, w.w_down, D, s.F);
    map(&L.m_kv, (const char*)w.w_qkv + (size_t)s.Dq * D * 2, 2 * s.Dkv, D);
    Epi e = epi0();
    e.kind = EPI_QKV; e.bias = w.b_qkv; e.out_t = s.q; e.ld_t = s.Dq;
    e.row_tok = s.row_tok[par]; e.tok_seq = s.tok_seq; e.tok_pos = s.tok_pos; e.cache = s.cache; e.layer0 = l;
    e.n_q_cols = s.Dq; e.n_kv_cols = s.Dkv; e.head_dim = s.dh; e.rope = s.family == ADEPT_FAMILY_LLAMA;
    e.rope_table = s.rope_table;
    L.e_qkv = e;
    e = epi0();
    e.kind = EPI_RESID; e.bias = w.b_o; e.out_f32 = s.X_out; e.ld_f32 = D; e.resid = s.X_in[par]; e.ld_resid = D;
    L.e_o = e;
    e = epi0();
    if (s.family == ADEPT_FAMILY_LLAMA) {
      e.kind = EPI_SWIGLU;
    } else {
      e.kind = EPI_ACT;
      e.act = ACT_GELU_TANH;
    }
    e.bias = w.b_up; e.out_t = s.hbuf; e.ld_t = s.F;
    L.e_up = e;
    e = epi0();
    e.kind = EPI_RESID; e.bias = w.b_down; e.out_f32 = s.X_out; e.ld_f32 = D; e.resid = s.X_out; e.ld_resid = D;
    L.e_down = e;
    e = epi0();
    e.kind = EPI_KV; e.bias = w.b_qkv + s.Dq; e.row_tok = s.exit_tok; e.tok_seq = s.tok_seq; e.tok_pos = s.tok_pos;
    e.cache = s.cache; e.layer0 = l; e.n_q_cols = 0; e.n_kv_cols = s.Dkv; e.head_dim = s.dh;
    e.rope = s.family == ADEPT_FAMILY_LLAMA; e.rope_table = s.rope_table;
    L.e_kv = e;
  }
  map(&h.m_h[0], s.hsm_w1, s.m1, D);
  map(&h.m_h[1], s.hsm_w2, s.m2, s.m1);
  map(&h.m_h[2], s.hsm_w3, s.m1, s.m2);
  map(&h.m_h[3], s.hsm_w4, D, s.m1);
  map(&h.m_head, s.w_head, s.V, D);
  if (!ok) {
    df_destroy(d);
    return no("tensor-map encoding failed");
  }
  {
    Epi e = epi0();
    e.kind = EPI_ACT; e.act = ACT_GELU_ERF; e.bias = s.hsm_b1; e.out_t = s.h1t; e.ld_t = s.m1; e.out_f32 = s.h1f;
    e.ld_f32 = s.m1;
    h.e_h[0] = e;
    e = epi0();
    e.kind = EPI_ACT; e.act = ACT_GELU_ERF; e.bias = s.hsm_b2; e.out_t = s.h2t; e.ld_t = s.m2;
    h.e_h[1] = e;
    e = epi0();
    e.kind = EPI_F32; e.bias = s.hsm_b3; e.out_f32 = s.h3f; e.ld_f32 = s.m1;
    h.e_h[2] = e;
    e = epi0();
    e.kind = EPI_F32; e.bias = s.hsm_b4; e.out_f32 = s.h5f; e.ld_f32 = D;
    h.e_h[3] = e;
    e = epi0();
    e.kind = EPI_F32; e.bias = s.b_head; e.out_f32 = s.logits; e.ld_f32 = s.V;
    h.e_head = e;
  }
  h.N = s.N; h.D = D; h.Dq = s.Dq; h.Dkv = s.Dkv; h.H = s.H; h.Hkv = s.Hkv; h.dh = s.dh; h.F = s.F;
  h.up_rows = s.L[0].up_rows; h.V = s.V; h.m1 = s.m1; h.m2 = s.m2; h.family = s.family; h.norm_mode = s.norm_mode;
  h.nqkv = nqkv; h.eps = s.eps; h.hsm_eps = s.hsm_eps; h.seq_cap = s.seq_cap; h.max_pos = s.max_pos;
  h.tok_emb = (const bf16*)s.tok_emb; h.pos_emb = (const bf16*)s.pos_emb;
  h.hsm_g0 = s.hsm_g0; h.hsm_conv = s.hsm_conv; h.hsm_g1 = s.hsm_g1; h.hsm_g2 = s.hsm_g2;
  h.cache = s.cache;
  for (int k = 0; k < 2; ++k) {
    h.X_in[k] = s.X_in[k];
    h.I[k] = s.I[k];
    h.row_tok[k] = s.row_tok[k];
  }
  h.X_out = s.X_out; h.tok_seq = s.tok_seq; h.tok_pos = s.tok_pos; h.seq_len = s.seq_len; h.ctr = s.ctr; h.err = s.err;
  h.q = (bf16*)s.q; h.att = (bf16*)s.att; h.hbuf = (bf16*)s.hbuf; h.xfill = (bf16*)s.xfill; h.h1t = (bf16*)s.h1t;
  h.h2t = (bf16*)s.h2t; h.hsm_s = s.hsm_s; h.hsm_prev = s.hsm_prev; h.hsm_I = s.hsm_I; h.final_ = s.final_;
  h.c0f = s.c0f; h.h1f = s.h1f; h.h3f = s.h3f; h.h5f = s.h5f; h.exit_tok = s.exit_tok;
  // workspaces
  h.lstride = (long long)s.cache.n_blocks * s.cache.n_kv_heads * s.cache.block_tokens * s.cache.head_dim;
  h.rope_table = s.family == ADEPT_FAMILY_LLAMA ? s.rope_table : nullptr;
  h.pool_elems = h.lstride * s.N;
  {
    const int bt = s.cache.block_tokens;
    h.bt_shift = (bt & (bt - 1)) == 0 ? __builtin_ctz((unsigned)bt) : -1;
  }
  d->lstride = h.lstride;
  void* p = nullptr;
  ok = true;
  ok = ok && dmalloc(d, &p, (size_t)kMaxB * s.H * kAttnMaxSplit * (s.dh + 2) * 4); h.attn_ws = (float*)p;
  ok = ok && dmalloc(d, &p, (size_t)kMaxB * s.H * 4); h.attn_cnt = (unsigned*)p;
  ok = ok && dmalloc(d, &p, (size_t)d->grid * kMaxB * 4); h.amax_v = (float*)p;
  ok = ok && dmalloc(d, &p, (size_t)d->grid * kMaxB * 4); h.amax_i = (int*)p;
  ok = ok && dmalloc(d, &p, 64); h.amax_cnt = (unsigned*)p;
  ok = ok && dmalloc(d, &p, 64); h.bar = (unsigned*)p;
  ok = ok && dmalloc(d, &p, 64); h.dbg = (unsigned*)p;
#ifdef ADEPT_DF_TRACE
  g_dbg_words = h.dbg;
#endif
  d->dlayers = ok ? (DfLayerDev*)arena_alloc(sizeof(DfLayerDev) * s.N) : nullptr;
  d->dplan = ok ? (DfPlan*)arena_alloc(sizeof(DfPlan)) : nullptr;
  ok = ok && d->dlayers && d->dplan;
  if (!ok) {
    df_destroy(d);
    return no("workspace allocation failed");
  }
  h.L = d->dlayers;
  if (cudaMemcpy(d->dlayers, hl.data(), sizeof(DfLayerDev) * s.N, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(d->dplan, &h, sizeof(DfPlan), cudaMemcpyHostToDevice) != cudaSuccess) {
    cudaGetLastError();
    df_destroy(d);
    return no("plan upload failed");
  }
  return d;
}

int df_max_batch(const DfState* d) { return d ? d->b_max : 0; }
int df_grid(const DfState* d) { return d ? d->grid : 0; }

cudaError_t df_step(DfState* d, cudaStream_t st, int B, const int* tokens, const int* forced, float delta,
                    int hsm_identity, const int* h_pos, int* exit_out, float* sim_out, int* next_out) {
  DfCall c;
  memset(&c, 0, sizeof c);
  c.P = d->dplan;
  c.tokens = tokens;
  c.forced = forced;
  c.delta = delta;
  c.B = B;
  c.identity = hsm_identity;
  c.exit_out = exit_out;
  c.sim_out = sim_out;
  c.next_out = next_out;
  c.ring = d->ring;
  c.x_bytes = d->x_bytes;
  c.rb = d->rb;
  c.lstride = d->lstride;
  int max_keys = 1;
  for (int b = 0; b < B; ++b) {
    c.pos[b] = h_pos[b];
    max_keys = std::max(max_keys, h_pos[b] + 1);
  }
  // key split: (rows x heads x splits) covers the consumer warps of the grid once
  const int warps = d->grid * kConsWarps;
  int nsplit = std::max(1, std::min(kAttnMaxSplit, (warps + B * d->H - 1) / (B * d->H)));
  int chunk = (std::max(max_keys, 1) + nsplit - 1) / nsplit;
  chunk = ((chunk + 31) / 32) * 32;
  nsplit = std::max(1, (max_keys + chunk - 1) / chunk);
  c.attn_chunk = chunk;
  c.attn_nsplit = nsplit;
  void* args[] = {&c};
  const cudaError_t e =
      cudaLaunchCooperativeKernel((const void*)df_kernel, dim3(d->grid), dim3(kThreads), args, (size_t)d->smem, st);
  return e;
}

void df_reset(DfState* d, cudaStream_t st) {
  if (!d) return;
  DfPlan h;
  if (cudaMemcpy(&h, d->dplan, sizeof h, cudaMemcpyDeviceToHost) != cudaSuccess) return;
  cudaMemsetAsync(h.bar, 0, 64, st);
  cudaMemsetAsync(h.amax_cnt, 0, 64, st);
}

}  // namespace adept

#ifdef ADEPT_DF_TRACE
extern "C" __attribute__((visibility("default"))) int adept_debug_df_prof(unsigned long long* out) {
  return cudaMemcpyFromSymbol(out, adept::g_df_prof, sizeof(unsigned long long) * 2 * 32) == cudaSuccess ? 0 : 1;
}
extern "C" __attribute__((visibility("default"))) int adept_debug_df_check(unsigned* out) {
  if (!adept::g_dbg_words) return 1;
  return cudaMemcpy(out, adept::g_dbg_words, 8, cudaMemcpyDeviceToHost) == cudaSuccess ? 0 : 1;
}
extern "C" __attribute__((visibility("default"))) int adept_debug_df_work(unsigned long long* out) {
  return cudaMemcpyFromSymbol(out, adept::g_df_work, sizeof(unsigned long long) * 256 * 16) == cudaSuccess ? 0 : 1;
}
#endif

// Prompt-pass attention on the tcgen05 tensor cores (sm_103a) over the paged KV cache.
//
// CTA = one tile of 128 active query rows x one head; 8 warps:
//   warps 0, 2      TMA producers: the Q tile once (2-D box of the pass's Q rows) and per
//                   128-key tile the sequence's 8 cache blocks of K (warp 0) and of V (warp 2)
//                   (one 16-row box per block and 64-wide half of the head), two stages each
//   warp 1          tensor-memory allocator; lane 0 issues S = Q K^T (M 128, N 128 keys, K d_h,
//                   both operands K-major) into one of two S accumulators, and O += P V (A = P
//                   from tensor memory, two buffers; B = the V tile as stored, MN-major) into the
//                   O accumulator, each as soon as its inputs are there
//   warps 4..11     softmax: two threads per query row (its TMEM lane), each with half of the
//                   keys; S by tcgen05.ld, masking (causal, the row's sequence, the keys present),
//                   online softmax in the exp2 domain (row maxima exchanged between the two),
//                   P rounded to bf16 into tensor memory; at the end O / l to the output, half
//                   of the columns each
// Tensor memory (512 columns): S 0-255 (two buffers), O 256-383, P 384-511 (two buffers).
// The running maximum of a row is raised only when a tile's maximum exceeds it by more than
// 2^8 (then the row of O is rescaled in TMEM); below that the probabilities stay <= 2^8, which
// bf16 and the fp32 accumulator carry exactly as well, and O / l is the same softmax.
// A tile of rows may span several sequences (rows are in sequence order): the key tiles of
// each sequence's run are processed in turn, the other rows' probabilities are zero there.
// Every mbarrier wait is bounded (the runtime wait limit); on time-out the CTA sets the error
// word, stops, drains its MMAs and copies and frees its tensor memory.
#define ADEPT_TU_ID 6
#include "attention_tc.h"
#include "gemm_tc.h"
#include "tc_ptx.cuh"

#include <cuda.h>

namespace adept {
namespace {

constexpr int AT_BM = 128;        // query rows per CTA
constexpr int AT_BN = 128;        // keys per tile
constexpr int AT_THREADS = 384;   // K producer, MMA, V producer, idle, 8 softmax warps (two per row)
constexpr int AT_MAX_SEG = 128;
constexpr float AT_RESCALE_LOG2 = 8.f;   // raise the running maximum only beyond 2^8
constexpr long long AT_DRAIN_CYCLES = 4000000000LL;

template <int DH>
struct AtLayout {
  static constexpr int HALVES = DH / 64;
  static constexpr int Q_BYTES = HALVES * AT_BM * 128;    // [half][row][128 B]
  static constexpr int KV_BYTES = HALVES * AT_BN * 128;   // one K or V stage: [half][key][128 B]
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + 2 * KV_BYTES;
  static constexpr int TOTAL = OFF_V + 2 * KV_BYTES;
};

struct AtParams {
  CUtensorMap qmap;   // Q rows [rows][ld_q], box {64, 128}
  CUtensorMap kmap;   // K pool as [layers * blocks * kv heads * 16][d_h], box {64, 16}
  CUtensorMap vmap;
  bf16* out;
  int ld_out;
  DevRange rows;
  const int* row_tok;
  const int* tok_seq;
  const int* tok_pos;
  const int* seq_len;
  const int* block_table;
  int max_blocks_per_seq, n_blocks, n_kv_heads, block_tokens;
  int layer0, n_heads, causal;
  float scale_log2;
  unsigned* err;
};

// Instruction descriptor, kind::f16: D fp32, A and B bf16, M = 128; b_mn: B is MN-major.
__device__ __forceinline__ constexpr uint32_t at_idesc(int n, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn ? (1u << 16) : 0u) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(128 >> 4) << 24);
}
// Shared-memory descriptor of an MN-major operand in 128-byte-swizzled atoms (64 MN elements x
// 8 K rows, 1024 bytes): lbo = bytes between 64-element MN chunks, K groups of 8 rows 1024 bytes
// apart.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFF);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])),
      "r"(__float_as_uint(v[11])), "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])),
      "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])),
      "r"(__float_as_uint(v[17])), "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])),
      "r"(__float_as_uint(v[20])), "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])),
      "r"(__float_as_uint(v[23])), "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])),
      "r"(__float_as_uint(v[26])), "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])),
      "r"(__float_as_uint(v[29])), "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// D[tmem] (+)= A[tmem] * B[smem], M = 128, K = 16: A's 128 rows in TMEM lanes, 2 bf16 per column.
__device__ __forceinline__ void umma_bf16_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\ntcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d),
      "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
// 64 consecutive fp32 columns of this thread's lane in one load.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, "
      "%38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, "
      "%60, %61, %62, %63}, [%64];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]),
        "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]),
        "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]),
        "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]),
        "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 64; ++j) v[j] = __uint_as_float(r[j]);
}
__device__ __forceinline__ void tmem_st32u(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
      "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
      "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
}
// 2^x by the hardware approximation (relative error ~2^-22; 0 for -inf): one instruction.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Non-blocking probe of a phase (try_wait may suspend the thread for a while; a loop that
// watches several barriers must not sit in one of them).
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// A bounded wait taken by every lane of a warp; the warp agrees on the outcome.
__device__ __forceinline__ bool at_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort_flag, unsigned* err,
                                             long long lim) {
  const bool ok = mbar_wait(bar, parity, abort_flag, err, lim);
  return __all_sync(0xffffffffu, ok) != 0;
}

template <int DH>
__global__ void __launch_bounds__(AT_THREADS, 1) attn_tc_kernel(const __grid_constant__ AtParams p) {
  using L = AtLayout<DH>;
  extern __shared__ __align__(1024) uint8_t at_raw[];
  __shared__ __align__(8) uint64_t q_full, k_full[2], v_full[2], k_empty[2], v_empty[2], s_full[2], s_free[2],
      p_full[2], pv_done[2], drain;
  __shared__ __align__(8) uint64_t pair_bar[4];   // the two softmax warps of a row quarter
  __shared__ float s_xch[2][2][AT_BM];              // their exchanged row maxima / sums
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ int s_rseq[AT_BM], s_rpos[AT_BM];
  __shared__ int s_seg_sq[AT_MAX_SEG], s_seg_kend[AT_MAX_SEG];
  __shared__ int s_nseg, s_nit;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const long long wlim = wait_limit();
  volatile int* abort_flag = &s_abort;
  uint8_t* sm = at_raw + ((1024 - (smem_u32(at_raw) & 1023)) & 1023);
  uint8_t* sQ = sm + L::OFF_Q;
  uint8_t* sK = sm + L::OFF_K;
  uint8_t* sV = sm + L::OFF_V;
  const int h = blockIdx.y, kvh = h / (p.n_heads / p.n_kv_heads);
  const int tile = (int)gridDim.x - 1 - (int)blockIdx.x;   // late (long causal) tiles start first

  if (tid == 0) {
    mbar_init(&q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_empty[s], 1);
      mbar_init(&s_full[s], 1);
      mbar_init(&s_free[s], 8);
    }
    mbar_init(&p_full[0], 8);
    mbar_init(&p_full[1], 8);
    for (int q = 0; q < 4; ++q) mbar_init(&pair_bar[q], 2);
    mbar_init(&pv_done[0], 1);
    mbar_init(&pv_done[1], 1);
    mbar_init(&drain, 1);
    s_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_wait();   // Q rows, row maps and the cache come from the preceding kernels
  pdl_launch_dependents();
  const int r0 = p.rows.b() + tile * AT_BM, rend = p.rows.e();
  if (r0 >= rend) return;   // uniform: no rows for this tile

  // rows of the tile: sequence and position (sequence -1 past the active range)
  if (tid < AT_BM) {
    const int r = r0 + tid;
    if (r < rend) {
      const int tok = p.row_tok[r];
      s_rseq[tid] = p.tok_seq[tok];
      s_rpos[tid] = p.tok_pos[tok];
    } else {
      s_rseq[tid] = -1;
      s_rpos[tid] = -1;
    }
  }
  if (warp == 1) {
    tmem_alloc(&s_tmem, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // runs of one sequence (rows are in sequence order) and each run's key range, in parallel:
  // thread = row; a run's index is the count of run starts up to its row
  __shared__ int s_wfirst[AT_BM / 32];
  bool first = false;
  unsigned bal = 0;
  if (tid < AT_BM) {
    const int sq = s_rseq[tid];
    first = sq >= 0 && (tid == 0 || s_rseq[tid - 1] != sq);
    bal = __ballot_sync(0xffffffffu, first);
    if (lane == 0) s_wfirst[warp] = __popc(bal);
  }
  __syncthreads();
  int g_row = -1;
  if (tid < AT_BM && s_rseq[tid] >= 0) {
    int before = 0;
    for (int w = 0; w < warp; ++w) before += s_wfirst[w];
    g_row = before + __popc(bal & ((2u << lane) - 1u)) - 1;
    if (first) {
      s_seg_sq[g_row] = s_rseq[tid];
      s_seg_kend[g_row] = 0;
    }
  }
  if (tid == 0) s_nseg = s_wfirst[0] + s_wfirst[1] + s_wfirst[2] + s_wfirst[3];
  __syncthreads();
  if (g_row >= 0) {
    const int sq = s_rseq[tid];
    const int kend = p.causal ? s_rpos[tid] + 1 : p.seq_len[sq];
    atomicMax(&s_seg_kend[g_row], min(kend, p.max_blocks_per_seq * p.block_tokens));
  }
  __syncthreads();
  if (warp == 0) {
    int n = 0;
    for (int g = lane; g < s_nseg; g += 32) n += (s_seg_kend[g] + AT_BN - 1) / AT_BN;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    if (lane == 0) s_nit = n;
  }
  __syncthreads();
  const int nseg = s_nseg, nit = s_nit;
  const uint32_t tmem = s_tmem;

  if (warp == 0 || warp == 2) {
    // ---- producers: warp 0 the Q tile and the K tiles, warp 2 the V tiles (K of a stage is
    // free once S of its previous tile is computed, V once O is, so K runs ahead of V); lane 0
    // issues, lanes 0..7 look up a tile's 8 cache blocks in parallel
    const bool kw = warp == 0;
    uint64_t* full = kw ? k_full : v_full;
    uint64_t* empty = kw ? k_empty : v_empty;
    const CUtensorMap* map = kw ? &p.kmap : &p.vmap;
    uint8_t* dst0 = kw ? sK : sV;
    int issued = 0;
    bool ok = true;
    if (kw && lane == 0) {
      mbar_expect_tx(&q_full, (uint32_t)L::Q_BYTES);
      for (int hf = 0; hf < L::HALVES; ++hf) tma_load_2d(&p.qmap, &q_full, sQ + hf * AT_BM * 128, h * DH + hf * 64, r0);
    }
    int it = 0;
    for (int g = 0; g < nseg && ok; ++g) {
      const int sq = s_seg_sq[g], kend = s_seg_kend[g];
      const int nt = (kend + AT_BN - 1) / AT_BN, nbv = (kend + 15) / 16;
      const int* bt = p.block_table + (size_t)sq * p.max_blocks_per_seq;
      for (int j = 0; j < nt && ok; ++j, ++it) {
        const int s = it & 1;
        int myrow = 0;
        if (lane < AT_BN / 16) {
          // blocks past the run's last key load the last block again (finite values; their
          // keys are masked and their V rows zeroed before use)
          int blk = bt[min(j * (AT_BN / 16) + lane, nbv - 1)];
          if (blk < 0 || blk >= p.n_blocks) {
            if (kw) atomicOr(p.err, ERRW_POS);
            blk = 0;
          }
          myrow = ((p.layer0 * p.n_blocks + blk) * p.n_kv_heads + kvh) * 16;
        }
        int rows8[AT_BN / 16];
#pragma unroll
        for (int b = 0; b < AT_BN / 16; ++b) rows8[b] = __shfl_sync(0xffffffffu, myrow, b);
        if (it >= 2 && !(ok = at_wait_warp(&empty[s], (uint32_t)(((it >> 1) - 1) & 1), abort_flag, p.err, wlim)))
          break;
        if (lane == 0) {
          mbar_expect_tx(&full[s], (uint32_t)L::KV_BYTES);
          for (int b = 0; b < AT_BN / 16; ++b)
            for (int hf = 0; hf < L::HALVES; ++hf)
              tma_load_2d(map, &full[s], dst0 + s * L::KV_BYTES + hf * AT_BN * 128 + b * 16 * 128, hf * 64, rows8[b]);
        }
        __syncwarp();
        issued = it + 1;
      }
    }
    // every copy issued has landed before the CTA ends (at most the last two tiles are open)
    if (lane == 0) {
      if (kw) {
        const long long tq = clock64();
        while (!mbar_try_wait(&q_full, 0) && clock64() - tq < AT_DRAIN_CYCLES) {
        }
      }
      for (int t = max(0, issued - 2); t < issued; ++t) {
        const long long t0 = clock64();
        while (!mbar_try_wait(&full[t & 1], (uint32_t)((t >> 1) & 1)) && clock64() - t0 < AT_DRAIN_CYCLES) {
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issue (lane 0); the whole warp zeroes V rows past a run's last key.  S of the
    // next tile and O of the current one are issued in whichever order their inputs arrive.
    constexpr uint32_t IDESC_S = at_idesc(AT_BN, false);
    constexpr uint32_t IDESC_O = at_idesc(DH, true);
    const uint32_t tO = tmem + 256;
    bool ok = at_wait_warp(&q_full, 0, abort_flag, p.err, wlim);
    tc_fence_after();
    auto issue_s = [&](int it) {
      const int s = it & 1;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t d = tmem + (uint32_t)(s * 128);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t a = sdesc_sw128(smem_u32(sQ + (kk >> 2) * AT_BM * 128) + (kk & 3) * 32);
          const uint64_t b = sdesc_sw128(smem_u32(sK + s * L::KV_BYTES + (kk >> 2) * AT_BN * 128) + (kk & 3) * 32);
          umma_bf16(d, a, b, IDESC_S, kk > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[s]);
        umma_commit(&k_empty[s]);
      }
      __syncwarp();
    };
    int ns = 0, npv = 0;   // next S and next O (P V) to issue
    int g = 0, j = 0;      // run and key tile of O npv
    long long idle0 = clock64();
    while (ok && npv < nit) {
      bool progress = false;
      if (ns < nit) {
        const int s = ns & 1;
        bool ready = mbar_test(&k_full[s], (uint32_t)((ns >> 1) & 1)) &&
                     (ns < 2 || mbar_test(&s_free[s], (uint32_t)(((ns >> 1) - 1) & 1)));
        ready = __shfl_sync(0xffffffffu, ready ? 1 : 0, 0) != 0;
        if (ready) {
          // every lane observes the completions before the tensor core reads the stage
          at_wait_warp(&k_full[s], (uint32_t)((ns >> 1) & 1), abort_flag, p.err, wlim);
          if (ns >= 2) at_wait_warp(&s_free[s], (uint32_t)(((ns >> 1) - 1) & 1), abort_flag, p.err, wlim);
          issue_s(ns);
          ++ns;
          progress = true;
        }
      }
      if (npv < ns) {
        const int s = npv & 1;
        bool ready = mbar_test(&p_full[s], (uint32_t)((npv >> 1) & 1)) &&
                     mbar_test(&v_full[s], (uint32_t)((npv >> 1) & 1));
        ready = __shfl_sync(0xffffffffu, ready ? 1 : 0, 0) != 0;
        if (ready) {
          at_wait_warp(&p_full[s], (uint32_t)((npv >> 1) & 1), abort_flag, p.err, wlim);
          at_wait_warp(&v_full[s], (uint32_t)((npv >> 1) & 1), abort_flag, p.err, wlim);
          const int nvalid = s_seg_kend[g] - j * AT_BN;
          if (nvalid < AT_BN) {
            // keys past the run's end: V rows may be unwritten memory; zero them (P is 0 there)
            uint8_t* v = sV + s * L::KV_BYTES;
            for (int hf = 0; hf < L::HALVES; ++hf)
              for (int c = nvalid * 8 + lane; c < AT_BN * 8; c += 32)
                *reinterpret_cast<uint4*>(v + hf * AT_BN * 128 + c * 16) = make_uint4(0, 0, 0, 0);
            fence_async_shared();
            __syncwarp();
          }
          tc_fence_after();
          if (lane == 0) {
            const uint32_t pa = tmem + 384 + (uint32_t)((npv & 1) * 64);   // P of this tile in TMEM
#pragma unroll
            for (int kk = 0; kk < AT_BN / 16; ++kk) {
              const uint64_t b = sdesc_mn_sw128(smem_u32(sV + s * L::KV_BYTES + kk * 16 * 128), (uint32_t)(AT_BN * 128));
              umma_bf16_ts(tO, pa + (uint32_t)(kk * 8), b, IDESC_O, (npv > 0 || kk > 0) ? 1u : 0u);
            }
            umma_commit(&pv_done[npv & 1]);
            umma_commit(&v_empty[s]);
          }
          __syncwarp();
          if (++j == (s_seg_kend[g] + AT_BN - 1) / AT_BN) {
            j = 0;
            ++g;
          }
          ++npv;
          progress = true;
        }
      }
      if (progress) {
        idle0 = clock64();
      } else if (!*abort_flag) {
        __nanosleep(32);   // leave the issue slots of this sub-partition to the softmax warps
      }
      if (progress) {
      } else if (*abort_flag) {
        ok = false;
      } else if (clock64() - idle0 > wlim) {
        if (lane == 0) atomicOr(p.err, ERRW_TIMEOUT);
        *abort_flag = 1;
        ok = false;
      }
      ok = __all_sync(0xffffffffu, ok) != 0;
    }
    // every MMA issued has completed before tensor memory is freed
    if (lane == 0) {
      umma_commit(&drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(&drain, 0) && clock64() - t0 < AT_DRAIN_CYCLES) {
      }
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---- softmax and output: two threads per query row (TMEM lane), each with half of the
    // tile's keys and half of O's columns; the pair exchanges its row maxima every tile (and
    // the sums once at the end) through shared memory, ordered by a bounded pair barrier
    const int q4 = (warp - 4) & 3, half = (warp - 4) >> 2;
    const int t = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    const int rsq = s_rseq[t], rpos = s_rpos[t];
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    int it = 0;
    constexpr int OC = DH / 64;   // 32-column chunks of O per thread
    auto pair_exchange = [&](float mine, int k) -> float {   // value of the partner thread
      s_xch[k & 1][half][t] = mine;
      __syncwarp();
      if (lane == 0) mbar_arrive(&pair_bar[q4]);
      if (!(ok = at_wait_warp(&pair_bar[q4], (uint32_t)(k & 1), abort_flag, p.err, wlim))) return mine;
      return s_xch[k & 1][half ^ 1][t];
    };
    for (int g = 0; g < nseg && ok; ++g) {
      const int sq = s_seg_sq[g], kend = s_seg_kend[g];
      const bool in_seg = rsq == sq;
      const int kend_r = in_seg ? (p.causal ? rpos + 1 : kend) : 0;
      const int nt = (kend + AT_BN - 1) / AT_BN;
      for (int j = 0; j < nt; ++j, ++it) {
        const int b = it & 1;
        if (!(ok = at_wait_warp(&s_full[b], (uint32_t)((it >> 1) & 1), abort_flag, p.err, wlim))) break;
        tc_fence_after();
        // two passes over this thread's 64 S columns: the maximum, then exp2, the sum and the
        // bf16 P; 8 partial chains
        const int nk = min(max(kend_r - j * AT_BN, 0), AT_BN);
        const uint32_t s_addr = tmem + lane_base + (uint32_t)(b * 128);
        const float sc = p.scale_log2;
        float mx[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) mx[q] = -INFINITY;
        // this thread's 64 columns in one load, kept in registers for both passes
        float sv[64];
        tmem_ld64(s_addr + (uint32_t)(half * 64), sv);
        const int k0 = half * 64;
#pragma unroll
        for (int e = 0; e < 64; ++e) {
          sv[e] = k0 + e < nk ? sv[e] * sc : -INFINITY;
          mx[e & 7] = fmaxf(mx[e & 7], sv[e]);
        }
        float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                           fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
        tmax = fmaxf(tmax, pair_exchange(tmax, it));
        if (!ok) break;
        float m_new = m;
        if (tmax > m && (m == -INFINITY || tmax - m > AT_RESCALE_LOG2)) m_new = tmax;
        const float factor = (m == -INFINITY || m_new == m) ? 1.f : exp2f(m - m_new);
        // masked keys take exp2(-inf) = 0; a row with no key here keeps m = -inf and takes 0
        const float mref = m_new == -INFINITY ? 0.f : m_new;
        // P's buffer (two in TMEM) is free once O of the tile before the previous one is done;
        // a rescale of O also needs O of the previous tile
        if (it >= 2 && !(ok = at_wait_warp(&pv_done[it & 1], (uint32_t)(((it >> 1) - 1) & 1), abort_flag, p.err, wlim)))
          break;
        const bool rescale = __any_sync(0xffffffffu, factor != 1.f) != 0;
        if (rescale && it >= 1 &&
            !(ok = at_wait_warp(&pv_done[(it - 1) & 1], (uint32_t)(((it - 1) >> 1) & 1), abort_flag, p.err, wlim)))
          break;
        tc_fence_after();
        if (rescale) {
#pragma unroll 1
          for (int c = half * OC; c < half * OC + OC; ++c) {
            float v[32];
            tmem_ld32(tmem + lane_base + (uint32_t)(256 + c * 32), v);
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= factor;
            tmem_st32(tmem + lane_base + (uint32_t)(256 + c * 32), v);
          }
          tmem_st_wait();
        }
        float sm[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) sm[q] = 0.f;
        uint32_t pk[32];
#pragma unroll
        for (int e = 0; e < 64; e += 2) {
          const float p0 = ex2_approx(sv[e] - mref);   // masked keys: exp2(-inf) = 0
          const float p1 = ex2_approx(sv[e + 1] - mref);
          sm[(e >> 1) & 7] += p0 + p1;
          const __nv_bfloat162 pr = __floats2bfloat162_rn(p0, p1);
          pk[e >> 1] = *reinterpret_cast<const uint32_t*>(&pr);
        }
        // this thread's keys -> P columns half*32 .. +31 of this tile's buffer (2 keys a column)
        tmem_st32u(tmem + lane_base + (uint32_t)(384 + (it & 1) * 64 + half * 32), pk);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[b]);   // S of this buffer is read
        const float rs = ((sm[0] + sm[1]) + (sm[2] + sm[3])) + ((sm[4] + sm[5]) + (sm[6] + sm[7]));
        l = l * factor + rs;   // this thread's keys; the pair's sums are added at the end
        m = m_new;
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[it & 1]);
      }
    }
    if (ok && nit > 0)
      ok = at_wait_warp(&pv_done[(nit - 1) & 1], (uint32_t)(((nit - 1) >> 1) & 1), abort_flag, p.err, wlim);
    if (ok) l += pair_exchange(l, it);
    tc_fence_after();
    const int r = r0 + t;
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
    for (int c = half * OC; c < half * OC + OC; ++c) {
      float v[32];
      tmem_ld32(tmem + lane_base + (uint32_t)(256 + c * 32), v);
      if (ok && rsq >= 0) {
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const __nv_bfloat162 pr = __floats2bfloat162_rn(v[2 * e] * inv, v[2 * e + 1] * inv);
          w[e] = *reinterpret_cast<const uint32_t*>(&pr);
        }
        uint4* o = reinterpret_cast<uint4*>(p.out + (size_t)r * p.ld_out + h * DH + c * 32);
#pragma unroll
        for (int e = 0; e < 4; ++e) o[e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

bool g_at_attr[2] = {false, false};

}  // namespace

int launch_attention_tc(cudaStream_t st, const void* q, int ld_q, int q_rows, void* out, int ld_out, DevRange rows,
                        int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos, const int* seq_len,
                        const KVCacheView& cache, int n_layers, int layer0, int n_heads, int causal, float scale_log2,
                        unsigned* err) {
  const int dh = cache.head_dim;
  if (!tc_gemm_supported() || (dh != 64 && dh != 128) || cache.block_tokens != 16 || rows.begin) return -1;
  if (n_heads % cache.n_kv_heads || ld_q % 8 || ld_out % 8 || ((uintptr_t)q & 15) || ((uintptr_t)out & 15)) return -1;
  if (max_rows <= 0) return 0;
  thread_local AtParams prm;   // one per host thread
  memset(&prm, 0, sizeof prm);
  const uint64_t pool_rows = (uint64_t)n_layers * cache.n_blocks * cache.n_kv_heads * 16;
  if (!tc_encode_2d(&prm.qmap, q, (uint64_t)n_heads * dh, (uint64_t)q_rows, (uint64_t)ld_q * 2, AT_BM)) return -1;
  if (!tc_encode_2d(&prm.kmap, cache.k, (uint64_t)dh, pool_rows, (uint64_t)dh * 2, 16)) return -1;
  if (!tc_encode_2d(&prm.vmap, cache.v, (uint64_t)dh, pool_rows, (uint64_t)dh * 2, 16)) return -1;
  prm.out = (bf16*)out;
  prm.ld_out = ld_out;
  prm.rows = rows;
  prm.row_tok = row_tok;
  prm.tok_seq = tok_seq;
  prm.tok_pos = tok_pos;
  prm.seq_len = seq_len;
  prm.block_table = cache.block_table;
  prm.max_blocks_per_seq = cache.max_blocks_per_seq;
  prm.n_blocks = cache.n_blocks;
  prm.n_kv_heads = cache.n_kv_heads;
  prm.block_tokens = cache.block_tokens;
  prm.layer0 = layer0;
  prm.n_heads = n_heads;
  prm.causal = causal;
  prm.scale_log2 = scale_log2;
  prm.err = err;
  const dim3 grid((max_rows + AT_BM - 1) / AT_BM, n_heads);
  cudaError_t e;
  if (dh == 128) {
    const size_t smem = AtLayout<128>::TOTAL + 1024;
    if (!g_at_attr[1]) {
      if (cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
          cudaSuccess)
        return -1;
      g_at_attr[1] = true;
    }
    e = launch_k(attn_tc_kernel<128>, grid, dim3(AT_THREADS), smem, st, prm);
  } else {
    const size_t smem = AtLayout<64>::TOTAL + 1024;
    if (!g_at_attr[0]) {
      if (cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
          cudaSuccess)
        return -1;
      g_at_attr[0] = true;
    }
    e = launch_k(attn_tc_kernel<64>, grid, dim3(AT_THREADS), smem, st, prm);
  }
  return e == cudaSuccess ? 1 : -1;
}

}  // namespace adept

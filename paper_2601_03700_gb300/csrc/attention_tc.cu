// Prompt-pass attention on the tcgen05 tensor cores (sm_103a) over the paged KV cache.
//
// CTA = one tile of 128 active query rows x one head; 8 warps:
//   warp 0 lane 0   TMA producer: the Q tile once (2-D box of the pass's Q rows), then per
//                   128-key tile the sequence's 8 cache blocks of K and of V (one 16-row box
//                   per block and 64-wide half of the head), two stages
//   warp 1          tensor-memory allocator; lane 0 issues S = Q K^T (M 128, N 128 keys, K d_h,
//                   both operands K-major) into one of two S accumulators, and O += P V (A = P
//                   from shared memory, K-major; B = the V tile as stored, MN-major) into the O
//                   accumulator; S of tile j+1 is issued before O of tile j
//   warps 4..7      softmax: thread = query row = TMEM lane; S row by tcgen05.ld, masking
//                   (causal, the row's sequence, the keys present), online softmax in the exp2
//                   domain, P rounded to bf16 into shared memory (128-byte swizzle); at the end
//                   O / l to the output
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
constexpr int AT_THREADS = 256;
constexpr int AT_MAX_SEG = 128;
constexpr float AT_RESCALE_LOG2 = 8.f;   // raise the running maximum only beyond 2^8
constexpr long long AT_DRAIN_CYCLES = 4000000000LL;

template <int DH>
struct AtLayout {
  static constexpr int HALVES = DH / 64;
  static constexpr int Q_BYTES = HALVES * AT_BM * 128;    // [half][row][128 B]
  static constexpr int KV_BYTES = HALVES * AT_BN * 128;   // one K or V stage: [half][key][128 B]
  static constexpr int P_BYTES = (AT_BN / 64) * AT_BM * 128;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + 2 * KV_BYTES;
  static constexpr int OFF_P = OFF_V + 2 * KV_BYTES;
  static constexpr int TOTAL = OFF_P + P_BYTES;
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
  __shared__ __align__(8) uint64_t q_full, k_full[2], v_full[2], kv_empty[2], s_full[2], s_free[2], p_full, o_done,
      drain;
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
  uint8_t* sP = sm + L::OFF_P;
  const int h = blockIdx.y, kvh = h / (p.n_heads / p.n_kv_heads);
  const int tile = (int)gridDim.x - 1 - (int)blockIdx.x;   // late (long causal) tiles start first

  if (tid == 0) {
    mbar_init(&q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&kv_empty[s], 1);
      mbar_init(&s_full[s], 1);
      mbar_init(&s_free[s], 4);
    }
    mbar_init(&p_full, 4);
    mbar_init(&o_done, 1);
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
  if (tid == 0) {
    // runs of one sequence (rows are in sequence order) and each run's key range
    int n = 0, nit = 0;
    for (int i = 0; i < AT_BM && s_rseq[i] >= 0; ++i) {
      const int sq = s_rseq[i];
      if (i == 0 || sq != s_rseq[i - 1]) {
        s_seg_sq[n] = sq;
        s_seg_kend[n] = 0;
        ++n;
      }
      const int kend = p.causal ? s_rpos[i] + 1 : p.seq_len[sq];
      s_seg_kend[n - 1] = max(s_seg_kend[n - 1], min(kend, p.max_blocks_per_seq * p.block_tokens));
    }
    for (int g = 0; g < n; ++g) nit += (s_seg_kend[g] + AT_BN - 1) / AT_BN;
    s_nseg = n;
    s_nit = nit;
  }
  __syncthreads();
  const int nseg = s_nseg, nit = s_nit;
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    // ---- producer
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      mbar_expect_tx(&q_full, (uint32_t)L::Q_BYTES);
      for (int hf = 0; hf < L::HALVES; ++hf) tma_load_2d(&p.qmap, &q_full, sQ + hf * AT_BM * 128, h * DH + hf * 64, r0);
      int it = 0;
      for (int g = 0; g < nseg && ok; ++g) {
        const int sq = s_seg_sq[g], kend = s_seg_kend[g];
        const int nt = (kend + AT_BN - 1) / AT_BN, nbv = (kend + 15) / 16;
        const int* bt = p.block_table + (size_t)sq * p.max_blocks_per_seq;
        for (int j = 0; j < nt && ok; ++j, ++it) {
          const int s = it & 1;
          if (it >= 2 && !(ok = mbar_wait(&kv_empty[s], (uint32_t)(((it >> 1) - 1) & 1), abort_flag, p.err, wlim)))
            break;
          mbar_expect_tx(&k_full[s], (uint32_t)L::KV_BYTES);
          mbar_expect_tx(&v_full[s], (uint32_t)L::KV_BYTES);
          for (int b = 0; b < AT_BN / 16; ++b) {
            const int bi = j * (AT_BN / 16) + b;
            // blocks past the run's last key load the last block again (finite values; their
            // keys are masked and their V rows zeroed before use)
            int blk = bt[min(bi, nbv - 1)];
            if (blk < 0 || blk >= p.n_blocks) {
              atomicOr(p.err, ERRW_POS);
              blk = 0;
            }
            const int row = ((p.layer0 * p.n_blocks + blk) * p.n_kv_heads + kvh) * 16;
            for (int hf = 0; hf < L::HALVES; ++hf) {
              tma_load_2d(&p.kmap, &k_full[s], sK + s * L::KV_BYTES + hf * AT_BN * 128 + b * 16 * 128, hf * 64, row);
              tma_load_2d(&p.vmap, &v_full[s], sV + s * L::KV_BYTES + hf * AT_BN * 128 + b * 16 * 128, hf * 64, row);
            }
          }
          issued = it + 1;
        }
      }
      // every copy issued has landed before the CTA ends (at most the last two tiles are open)
      const long long tq = clock64();
      while (!mbar_try_wait(&q_full, 0) && clock64() - tq < AT_DRAIN_CYCLES) {
      }
      for (int t = max(0, issued - 2); t < issued; ++t) {
        const uint32_t ph = (uint32_t)((t >> 1) & 1);
        const long long t0 = clock64();
        while (!mbar_try_wait(&k_full[t & 1], ph) && clock64() - t0 < AT_DRAIN_CYCLES) {
        }
        while (!mbar_try_wait(&v_full[t & 1], ph) && clock64() - t0 < AT_DRAIN_CYCLES) {
        }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issue (lane 0); the whole warp zeroes V rows past a run's last key
    constexpr uint32_t IDESC_S = at_idesc(AT_BN, false);
    constexpr uint32_t IDESC_O = at_idesc(DH, true);
    const uint32_t tO = tmem + 256;
    bool ok = at_wait_warp(&q_full, 0, abort_flag, p.err, wlim);
    tc_fence_after();
    auto issue_s = [&](int it) -> bool {
      const int s = it & 1;
      if (!at_wait_warp(&k_full[s], (uint32_t)((it >> 1) & 1), abort_flag, p.err, wlim)) return false;
      if (it >= 2 && !at_wait_warp(&s_free[s], (uint32_t)(((it >> 1) - 1) & 1), abort_flag, p.err, wlim)) return false;
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
      }
      __syncwarp();
      return true;
    };
    if (ok && nit > 0) ok = issue_s(0);
    int g = 0, j = 0;   // run and key tile of iteration it
    for (int it = 0; it < nit && ok; ++it) {
      if (it + 1 < nit && !(ok = issue_s(it + 1))) break;
      const int s = it & 1;
      if (!(ok = at_wait_warp(&p_full, (uint32_t)(it & 1), abort_flag, p.err, wlim))) break;
      if (!(ok = at_wait_warp(&v_full[s], (uint32_t)((it >> 1) & 1), abort_flag, p.err, wlim))) break;
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
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk) {
          const uint64_t a = sdesc_sw128(smem_u32(sP + (kk >> 2) * AT_BM * 128) + (kk & 3) * 32);
          const uint64_t b = sdesc_mn_sw128(smem_u32(sV + s * L::KV_BYTES + kk * 16 * 128), (uint32_t)(AT_BN * 128));
          umma_bf16(tO, a, b, IDESC_O, (it > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&o_done);
        umma_commit(&kv_empty[s]);
      }
      __syncwarp();
      if (++j == (s_seg_kend[g] + AT_BN - 1) / AT_BN) {
        j = 0;
        ++g;
      }
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
    // ---- softmax and output: thread = query row = TMEM lane
    const int t = tid - 128;
    const uint32_t lane_base = (uint32_t)((warp - 4) * 32) << 16;
    const int rsq = s_rseq[t], rpos = s_rpos[t];
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    int it = 0;
    for (int g = 0; g < nseg && ok; ++g) {
      const int sq = s_seg_sq[g], kend = s_seg_kend[g];
      const bool in_seg = rsq == sq;
      const int kend_r = in_seg ? (p.causal ? rpos + 1 : kend) : 0;
      const int nt = (kend + AT_BN - 1) / AT_BN;
      for (int j = 0; j < nt; ++j, ++it) {
        const int b = it & 1;
        if (!(ok = at_wait_warp(&s_full[b], (uint32_t)((it >> 1) & 1), abort_flag, p.err, wlim))) break;
        tc_fence_after();
        float sv[AT_BN];
#pragma unroll
        for (int c = 0; c < AT_BN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_base + (uint32_t)(b * 128 + c * 32), v);
#pragma unroll
          for (int e = 0; e < 32; ++e) sv[c * 32 + e] = v[e];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[b]);
        const int nk = min(max(kend_r - j * AT_BN, 0), AT_BN);
        float tmax = -INFINITY;
#pragma unroll
        for (int c = 0; c < AT_BN; ++c)
          if (c < nk) tmax = fmaxf(tmax, sv[c] * p.scale_log2);
        float m_new = m;
        if (tmax > m && (m == -INFINITY || tmax - m > AT_RESCALE_LOG2)) m_new = tmax;
        const float factor = (m == -INFINITY || m_new == m) ? 1.f : exp2f(m - m_new);
        float rs = 0.f;
        uint32_t pk[AT_BN / 2];
#pragma unroll
        for (int c = 0; c < AT_BN; c += 2) {
          const float p0 = c < nk ? exp2f(sv[c] * p.scale_log2 - m_new) : 0.f;
          const float p1 = c + 1 < nk ? exp2f(sv[c + 1] * p.scale_log2 - m_new) : 0.f;
          rs += p0 + p1;
          const __nv_bfloat162 pr = __floats2bfloat162_rn(p0, p1);
          pk[c >> 1] = *reinterpret_cast<const uint32_t*>(&pr);
        }
        l = l * factor + rs;
        m = m_new;
        // O of the previous tile is complete (and P's buffer free) before it is rescaled or
        // P is rewritten
        if (it >= 1 && !(ok = at_wait_warp(&o_done, (uint32_t)((it - 1) & 1), abort_flag, p.err, wlim))) break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, factor != 1.f)) {
#pragma unroll
          for (int c = 0; c < DH / 32; ++c) {
            float v[32];
            tmem_ld32(tmem + lane_base + (uint32_t)(256 + c * 32), v);
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= factor;
            tmem_st32(tmem + lane_base + (uint32_t)(256 + c * 32), v);
          }
          tmem_st_wait();
        }
        // P row (bf16) into the K-major 128-byte-swizzled tile: half, then row, then 16-byte chunk
#pragma unroll
        for (int c8 = 0; c8 < AT_BN / 8; ++c8) {
          const int hf = c8 >> 3, ch = c8 & 7;
          uint8_t* dst = sP + hf * AT_BM * 128 + t * 128 + ((ch ^ (t & 7)) << 4);
          *reinterpret_cast<uint4*>(dst) = make_uint4(pk[c8 * 4], pk[c8 * 4 + 1], pk[c8 * 4 + 2], pk[c8 * 4 + 3]);
        }
        fence_async_shared();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full);
      }
    }
    if (ok && nit > 0) ok = at_wait_warp(&o_done, (uint32_t)((nit - 1) & 1), abort_flag, p.err, wlim);
    tc_fence_after();
    const int r = r0 + t;
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
    for (int c = 0; c < DH / 32; ++c) {
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

// Attention of the active query rows over the paged KV cache of one layer.  The keys
// of a sequence at layer i are every cached position of that layer -- computed by the
// token itself if it was active at i, or filled from its mapped state s~_N if it
// exited earlier -- so attention needs no knowledge of exits.
#include "common.cuh"
#include "kernels.h"

namespace adept {

// One warp per (query row, head); lanes own keys for the scores and head dimensions
// for the value sum; online softmax over blocks of 32 keys.
template <typename T, int DH>
__global__ void __launch_bounds__(256) attn_warp_kernel(const T* __restrict__ q, int ld_q, T* __restrict__ out,
                                                        int ld_out, DevRange rows, const int* row_tok,
                                                        const int* tok_seq, const int* tok_pos, const int* seq_len,
                                                        KVCacheView cache, int layer0, int n_heads, int causal,
                                                        float scale) {
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

template <typename T>
static void attn_dispatch(cudaStream_t st, const void* q, int ld_q, void* out, int ld_out, DevRange rows,
                          int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos,
                          const int* seq_len, KVCacheView cache, int layer0, int n_heads, int causal) {
  const int dh = cache.head_dim;
  const float scale = 1.f / sqrtf((float)dh);
  const int grid = cdiv(max_rows * n_heads, 8);
#define ATT_CASE(D)                                                                                         \
  case D:                                                                                                   \
    attn_warp_kernel<T, D><<<grid, 256, 0, st>>>((const T*)q, ld_q, (T*)out, ld_out, rows, row_tok, tok_seq, \
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

void launch_attention(cudaStream_t st, int dt, const void* q, int ld_q, void* out, int ld_out, DevRange rows,
                      int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos, const int* seq_len,
                      KVCacheView cache, int layer0, int n_heads, int causal) {
  if (max_rows <= 0) return;
  if (dt == 1)
    attn_dispatch<bf16>(st, q, ld_q, out, ld_out, rows, max_rows, row_tok, tok_seq, tok_pos, seq_len, cache, layer0,
                        n_heads, causal);
  else
    attn_dispatch<float>(st, q, ld_q, out, ld_out, rows, max_rows, row_tok, tok_seq, tok_pos, seq_len, cache, layer0,
                         n_heads, causal);
}

}  // namespace adept

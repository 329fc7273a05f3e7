// Row-wise kernels of the early-exit pass: embedding, norms, the exit test with
// active-token compaction, the HSM's non-GEMM steps, argmax, skipped-layer-fill
// bucketing and load-time weight repacking.
#define ADEPT_TU_ID 3
#include "common.cuh"
#include "kernels.h"

#include <math.h>

#include <algorithm>

namespace adept {

// ---------------------------------------------------------------------------
// pass set-up: token -> (sequence, position), identity row map, counters
// ---------------------------------------------------------------------------
__global__ void pass_init_kernel(int n_tok, int prompt_len, int decode, int* tok_seq, int* tok_pos,
                                 int* row_tok, int* seq_len, int seq_cap, int max_pos, unsigned* err, int* ctr,
                                 int n_ctr, float* sim, int n_layers, int* tok_exit) {
  PDL_ENTRY();
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  // the pass's counters: all active, nothing exited
  if (t < n_ctr) ctr[t] = t == CTR_ACTIVE ? n_tok : 0;
  if (t >= n_tok) return;
  // every token active: its exit layer so far is N
  if (tok_exit) tok_exit[t] = n_layers;
  // similarities not tested stay NaN
  if (sim)
    for (int l = 0; l < n_layers; ++l) sim[(size_t)t * n_layers + l] = __int_as_float(0x7fffffff);
  int s, p;
  if (decode) {
    s = t;
    p = seq_len[t];
    seq_len[t] = p + 1;
  } else {
    s = t / prompt_len;
    p = t % prompt_len;
    if (p == 0) seq_len[s] = prompt_len;
  }
  if (p >= seq_cap || (max_pos > 0 && p >= max_pos)) {
    atomicOr(err, ERRW_POS);
    p = 0;
  }
  tok_seq[t] = s;
  tok_pos[t] = p;
  row_tok[t] = t;
}

// ---------------------------------------------------------------------------
// embedding (s_0): token embedding (+ learned position) (+ type and LayerNorm for BERT)
// ---------------------------------------------------------------------------
// xhat (optional, decoders): each embedded row standardised for the first layer's
// attention input (smode, seps), as the standardisation kernel computes it, in bf16.
template <typename T>
__global__ void embed_kernel(const int* tokens, int n_tok, const int* tok_pos, const T* E, const T* P,
                             const float* type_emb, const float* g, const float* b, int family, int D, int V,
                             float eps, float* X, unsigned* err, bf16* xhat, int smode, float seps) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int t = blockIdx.x;
  if (t >= n_tok) return;
  int tok = tokens[t];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERRW_TOKEN);
    tok = 0;
  }
  const int pos = tok_pos[t];
  float* x = X + (size_t)t * D;
  float s1 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    float v = to_f(E[(size_t)tok * D + d]);
    if (P) v += to_f(P[(size_t)pos * D + d]);
    if (type_emb) v += type_emb[d];
    x[d] = v;
    s1 += v;
  }
  if (family != 2) {
    if (!xhat) return;
    // the thread re-reads only the elements it wrote
    const float mu = smode == NORM_LN ? block_sum(s1, red) / D : 0.f;
    float s2 = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      const float c = x[d] - mu;
      s2 += c * c;
    }
    const float tot = block_sum(s2, red);
    const float rs = smode == NORM_COPY ? 1.f : rsqrtf(tot / D + seps);
    const float m0 = smode == NORM_COPY ? 0.f : mu;
    for (int d = threadIdx.x; d < D; d += blockDim.x) xhat[(size_t)t * D + d] = __float2bfloat16_rn((x[d] - m0) * rs);
    return;
  }
  const float mu = block_sum(s1, red) / D;
  float s2 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float c = x[d] - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(block_sum(s2, red) / D + eps);
  for (int d = threadIdx.x; d < D; d += blockDim.x) x[d] = (x[d] - mu) * rstd * g[d] + b[d];
}

// Grid of the row kernels whose live row count is a device value, usually far below its
// bound in a prompt pass (the mapper's rows, the standardisation, the exit moves): the rows are
// taken in turn by at most per_sm CTAs per SM, so a pass whose bound is thousands of rows does
// not launch thousands of CTAs that find no row.
static int row_grid(int max_rows, int per_sm) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
  }
  return std::min(max_rows, per_sm * sms);
}
static int hsm_grid(int max_rows) { return row_grid(max_rows, 2); }

// ---------------------------------------------------------------------------
// standardisation of a layer input (gains folded into the next GEMM)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void standardize_kernel(const float* X, int ldx, const int* in_rows, DevRange rows, int D, int mode,
                                   float eps, T* out, int ld_out) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int rb = rows.b(), re = rows.e();
  for (int r = rb + blockIdx.x; r < re; r += gridDim.x) {   // rows of the live range, in turn
  const int src = in_rows ? in_rows[r] : r;
  const float* x = X + (size_t)src * ldx;
  T* o = out + (size_t)r * ld_out;
  if (mode == NORM_COPY) {
    for (int d = threadIdx.x; d < D; d += blockDim.x) o[d] = from_f<T>(x[d]);
    continue;
  }
  float mu = 0.f;
  if (mode == NORM_LN) {
    float s = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s += x[d];
    mu = block_sum(s, red) / D;
  }
  float s2 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float c = x[d] - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(block_sum(s2, red) / D + eps);
  for (int d = threadIdx.x; d < D; d += blockDim.x) o[d] = from_f<T>((x[d] - mu) * rstd);
  }
}

// In-place LayerNorm with gain and shift (the post-LN encoder's residual stream).
__global__ void layernorm_inplace_kernel(float* X, DevRange rows, int D, const float* g, const float* b, float eps) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int r = rows.b() + blockIdx.x;
  if (r >= rows.e()) return;
  float* x = X + (size_t)r * D;
  float s = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) s += x[d];
  const float mu = block_sum(s, red) / D;
  float s2 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float c = x[d] - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(block_sum(s2, red) / D + eps);
  for (int d = threadIdx.x; d < D; d += blockDim.x) x[d] = (x[d] - mu) * rstd * g[d] + b[d];
}

// ---------------------------------------------------------------------------
// exit test (Sec. 4.1): c = <s_i, I> / (|s_i| |I|) vs delta, or the forced layer
// ---------------------------------------------------------------------------

__global__ void exit_decide_kernel(const float* Xout, const float* I, const float* Xin, int D, DevRange rows,
                                   const int* row_tok, const int* forced, int layer, int n_layers,
                                   const float* delta_p, int test, int metric, float* sim, int* flag,
                                   float* inv_norm, unsigned* err) {
  PDL_ENTRY();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int r = warp;
  if (r >= rows.e()) return;
  const float* s = Xout + (size_t)r * D;
  const float* in = I + (size_t)r * D;
  const float* sp = Xin + (size_t)r * D;
  float ns = 0.f, ni = 0.f, dot = 0.f, np_ = 0.f, dp = 0.f;
  for (int d = lane; d < D; d += 32) {
    const float a = s[d], c = in[d];
    ns += a * a;
    ni += c * c;
    dot += a * c;
    if (metric != EXIT_GLOBAL) {
      const float b = sp[d];
      np_ += b * b;
      dp += a * b;
    }
  }
  ns = warp_sum(ns);
  ni = warp_sum(ni);
  dot = warp_sum(dot);
  np_ = warp_sum(np_);
  dp = warp_sum(dp);
  if (lane != 0) return;
  const int tok = row_tok[r];
  int ex = 0;
  if (test) {
    const float c = exit_similarity(metric, ns, ni, dot, np_, dp);
    if (sim) sim[(size_t)tok * n_layers + (layer - 1)] = c;
    const int f = forced ? forced[tok] : 0;
    if (f != 0 && (f < 2 || f > n_layers)) atomicOr(err, ERRW_FORCED);
    ex = (f > 0) ? (f == layer) : (c >= *delta_p);
  }
  flag[r] = ex;
  inv_norm[r] = ns > 0.f ? rsqrtf(ns) : 0.f;
}

// Single-CTA stable compaction of the active rows: survivors keep their order in the
// next active list; exits are appended to the pass's exit list.  Counter layout:
// ctr[CTR_ACTIVE + parity] active counts, ctr[CTR_EXITED] exits so far,
// ctr[CTR_PREFIX + i] exits after layer i.
__global__ void exit_scan_kernel(int* ctr, int in_parity, const int* flag, const int* row_tok, int* row_tok_next,
                                 int* exit_tok, int* dst, int* exit_layer_out, int layer, int aao_len,
                                 const int* tok_pos) {
  PDL_ENTRY();
  __shared__ int s_stay[1024];
  __shared__ int s_exit[1024];
  const int n = ctr[CTR_ACTIVE + in_parity];
  const int base = ctr[CTR_EXITED];
  const int tid = threadIdx.x, nt = blockDim.x;
  const int per = (n + nt - 1) / nt;
  const int lo = min(n, tid * per), hi = min(n, lo + per);
  // all-at-once (aao_len = prompt length): a row takes the decision of its sequence's last
  // prompt token, which is active with it at the same row offset (sequences stay whole)
  auto fl = [&](int r) {
    return aao_len ? flag[min(n - 1, r + (aao_len - 1 - tok_pos[row_tok[r]]))] : flag[r];
  };
  int ce = 0;
  for (int r = lo; r < hi; ++r) ce += fl(r);
  s_exit[tid] = ce;
  s_stay[tid] = (hi - lo) - ce;
  __syncthreads();
  for (int off = 1; off < nt; off <<= 1) {
    int a = 0, b = 0;
    if (tid >= off) {
      a = s_exit[tid - off];
      b = s_stay[tid - off];
    }
    __syncthreads();
    s_exit[tid] += a;
    s_stay[tid] += b;
    __syncthreads();
  }
  int e = s_exit[tid] - ce;
  int s = s_stay[tid] - ((hi - lo) - ce);
  for (int r = lo; r < hi; ++r) {
    const int tok = row_tok[r];
    if (fl(r)) {
      dst[r] = -1 - (base + e);
      exit_tok[base + e] = tok;
      if (exit_layer_out) exit_layer_out[tok] = layer;
      ++e;
    } else {
      dst[r] = s;
      row_tok_next[s] = tok;
      ++s;
    }
  }
  if (tid == nt - 1) {
    const int E = s_exit[nt - 1];
    ctr[CTR_ACTIVE + (in_parity ^ 1)] = s_stay[nt - 1];
    ctr[CTR_EXITED] = base + E;
    ctr[CTR_PREFIX + layer] = base + E;
  }
}

// Moves each active row to its new place: survivors -> next layer input (s_i) and the
// inertia with s_hat_i added (Sec. 4.1, after the test); exits -> the HSM input slots
// (s_i, s_{i-1}, inertia before s_hat_i).  first != 0 (layer 1): the inertia starts
// as s_hat_1 (the sum over earlier layers is empty).
__global__ void exit_move_kernel(const float* Xin, const float* Xout, const float* I, int first, int D,
                                 const int* n_rows, const int* dst, const float* inv_norm, float* Xnext, float* Inext,
                                 float* hsm_s, float* hsm_prev, float* hsm_I) {
  PDL_ENTRY();
  const int n = *n_rows;
  for (int r = blockIdx.x; r < n; r += gridDim.x) {
  const int d0 = dst[r];
  const float* s = Xout + (size_t)r * D;
  const float* in = I + (size_t)r * D;
  if (d0 >= 0) {
    const float w = inv_norm[r];
    float* xn = Xnext + (size_t)d0 * D;
    float* inn = Inext + (size_t)d0 * D;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      const float v = s[d];
      xn[d] = v;
      inn[d] = (first ? 0.f : in[d]) + v * w;
    }
  } else {
    const size_t k = (size_t)(-1 - d0);
    const float* sp = Xin + (size_t)r * D;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      hsm_s[k * D + d] = s[d];
      hsm_prev[k * D + d] = sp[d];
      hsm_I[k * D + d] = in[d];
    }
  }
  }
}

// The three steps above in one CTA, for passes with at most EXIT_SMALL_MAX active rows
// (generation steps): the similarity test, the stable compaction and the row moves.
__global__ void __launch_bounds__(256) exit_small_kernel(const float* Xin, const float* Xout, const float* I,
                                                         int first, int D, int* ctr, int par, const int* row_tok,
                                                         int* row_tok_next, const int* forced, int layer,
                                                         int n_layers, const float* delta_p, int test, float* sim,
                                                         int* exit_tok, int* exit_layer_out, float* Xnext,
                                                         float* Inext, float* hsm_s, float* hsm_prev, float* hsm_I,
                                                         int metric, int aao_len, const int* tok_pos,
                                                         unsigned* err) {
  PDL_ENTRY();
  __shared__ int s_dst[EXIT_SMALL_MAX];
  __shared__ float s_w[EXIT_SMALL_MAX];
  const int n = min(ctr[CTR_ACTIVE + par], EXIT_SMALL_MAX);
  const int base = ctr[CTR_EXITED];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const float delta = *delta_p;
  for (int r = warp; r < n; r += nw) {
    const float* s = Xout + (size_t)r * D;
    const float* in = I + (size_t)r * D;
    const float* sp = Xin + (size_t)r * D;
    float ns = 0.f, ni = 0.f, dot = 0.f, np_ = 0.f, dp = 0.f;
    for (int d = lane; d < D; d += 32) {
      const float a = s[d], c = in[d];
      ns += a * a;
      ni += c * c;
      dot += a * c;
      if (metric != EXIT_GLOBAL) {
        const float b = sp[d];
        np_ += b * b;
        dp += a * b;
      }
    }
    ns = warp_sum(ns);
    ni = warp_sum(ni);
    dot = warp_sum(dot);
    np_ = warp_sum(np_);
    dp = warp_sum(dp);
    if (lane == 0) {
      const int tok = row_tok[r];
      int ex = 0;
      if (test) {
        const float c = exit_similarity(metric, ns, ni, dot, np_, dp);
        if (sim) sim[(size_t)tok * n_layers + (layer - 1)] = c;
        const int f = forced ? forced[tok] : 0;
        if (f != 0 && (f < 2 || f > n_layers)) atomicOr(err, ERRW_FORCED);
        ex = (f > 0) ? (f == layer) : (c >= delta);
      }
      s_dst[r] = ex;
      s_w[r] = ns > 0.f ? rsqrtf(ns) : 0.f;
    }
  }
  __syncthreads();
  KT_MARK(0);
  if (threadIdx.x == 0) {
    int e = 0, k = 0;
    for (int r = 0; r < n; ++r) {
      const int tok = row_tok[r];
      // all-at-once: the decision of the sequence's last prompt token, a later row not yet
      // rewritten by this loop
      const int rl = aao_len ? min(n - 1, r + (aao_len - 1 - tok_pos[tok])) : r;
      if (s_dst[rl]) {
        s_dst[r] = -1 - (base + e);
        exit_tok[base + e] = tok;
        if (exit_layer_out) exit_layer_out[tok] = layer;
        ++e;
      } else {
        s_dst[r] = k;
        row_tok_next[k] = tok;
        ++k;
      }
    }
    ctr[CTR_ACTIVE + (par ^ 1)] = k;
    ctr[CTR_EXITED] = base + e;
    ctr[CTR_PREFIX + layer] = base + e;
  }
  __syncthreads();
  KT_MARK(1);
  for (int r = warp; r < n; r += nw) {
    const int d0 = s_dst[r];
    const float* s = Xout + (size_t)r * D;
    const float* in = I + (size_t)r * D;
    if (d0 >= 0) {
      const float w = s_w[r];
      float* xn = Xnext + (size_t)d0 * D;
      float* inn = Inext + (size_t)d0 * D;
      for (int d = lane; d < D; d += 32) {
        const float v = s[d];
        xn[d] = v;
        inn[d] = (first ? 0.f : in[d]) + v * w;
      }
    } else {
      const size_t kk = (size_t)(-1 - d0);
      const float* sp = Xin + (size_t)r * D;
      for (int d = lane; d < D; d += 32) {
        hsm_s[kk * D + d] = s[d];
        hsm_prev[kk * D + d] = sp[d];
        hsm_I[kk * D + d] = in[d];
      }
    }
  }
}

// The same test, compaction and moves for a generation step of at most 16 rows, in one
// pass over memory: each row's s_i, inertia and s_{i-1} are read once into registers (a
// row per 512 >> rshift threads), the decision and compaction run on the reduced sums,
// and the moves are written from the registers.
constexpr int EXD_THREADS = 512;
constexpr int EXD_V = 4;   // most float4 per thread per row vector
// V: float4 per thread per row vector, the fewest that cover a row (the kernel runs cold in
// every layer of a generation step, so its unrolled code is kept to what the rows need)
template <int V>
__global__ void __launch_bounds__(EXD_THREADS)
    exit_decode_kernel(const float* __restrict__ Xin, const float* __restrict__ Xout, const float* __restrict__ I,
                       int first, int D, int* ctr, int par, const int* row_tok, int* row_tok_next, const int* forced,
                       int layer, int n_layers, const float* delta_p, int test, float* sim, int* exit_tok,
                       int* exit_layer_out, float* __restrict__ Xnext, float* __restrict__ Inext,
                       float* __restrict__ hsm_s, float* __restrict__ hsm_prev, float* __restrict__ hsm_I, int rshift,
                       int max_rows, bf16* xhat_next, int smode, float seps, int metric, int aao_len,
                       const int* tok_pos, unsigned* err) {
  // Before the grid-dependency wait: everything the previous layer's exit kernel wrote (the
  // counters, the row map, the inertia and the layer input s_{i-1}), which has completed by the
  // time this kernel starts (the attention kernel between them releases its dependents only
  // after its own wait); after it: the layer output s_i.
  KT_BEGIN();
  __shared__ float s_red[EXD_THREADS / 32][6];
  __shared__ float s_mu[16];
  __shared__ int s_dst[16], s_tok[16];
  __shared__ float s_w[16];
  const int tpr = EXD_THREADS >> rshift;   // threads per row
  const int row = threadIdx.x >> (9 - rshift), sub = threadIdx.x & (tpr - 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // every independent load first: the counters, the decider's token and threshold, and the
  // row vectors of every row slot below the pass's row bound (slots past the active count
  // read rows of the pass's buffers whose values go unused)
  const int n = min(min(ctr[CTR_ACTIVE + par], 1 << rshift), max_rows);
  const int base = ctr[CTR_EXITED];
  const int tok_r = (int)threadIdx.x < max_rows ? row_tok[threadIdx.x] : 0;
  const int forced_r = forced && (int)threadIdx.x < max_rows ? forced[tok_r] : 0;   // the decider's forced layer
  const float delta = *delta_p;
  const int D4 = D >> 2;
  float4 xs[V], xi[V], xp[V];
  float ns = 0.f, ni = 0.f, dot = 0.f, sx = 0.f, np_ = 0.f, dp = 0.f;
  if (row < max_rows) {
    const float4* i4 = reinterpret_cast<const float4*>(I + (size_t)row * D);
    const float4* p4 = reinterpret_cast<const float4*>(Xin + (size_t)row * D);
#pragma unroll
    for (int j = 0; j < V; ++j) {
      const int v = sub + j * tpr;
      if (v < D4) {
        xi[j] = first ? make_float4(0.f, 0.f, 0.f, 0.f) : i4[v];
        xp[j] = p4[v];
      }
    }
  }
  pdl_wait();
  KT_WAITED();
  pdl_launch_dependents();
  if (row < max_rows) {
    const float4* s4 = reinterpret_cast<const float4*>(Xout + (size_t)row * D);
#pragma unroll
    for (int j = 0; j < V; ++j) {
      const int v = sub + j * tpr;
      if (v < D4) xs[j] = s4[v];
    }
#pragma unroll
    for (int j = 0; j < V; ++j) {
      if (row < n && sub + j * tpr < D4) {
        const float4 a = xs[j], c = xi[j];
        ns += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
        ni += c.x * c.x + c.y * c.y + c.z * c.z + c.w * c.w;
        dot += a.x * c.x + a.y * c.y + a.z * c.z + a.w * c.w;
        sx += a.x + a.y + a.z + a.w;
        const float4 b = xp[j];
        np_ += b.x * b.x + b.y * b.y + b.z * b.z + b.w * b.w;
        dp += a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w;
      }
    }
  }
  ns = warp_sum(ns);
  ni = warp_sum(ni);
  dot = warp_sum(dot);
  sx = warp_sum(sx);
  np_ = warp_sum(np_);
  dp = warp_sum(dp);
  if (lane == 0) {
    s_red[warp][0] = ns;
    s_red[warp][1] = ni;
    s_red[warp][2] = dot;
    s_red[warp][3] = sx;
    s_red[warp][4] = np_;
    s_red[warp][5] = dp;
  }
  __syncthreads();
  const int wpr = tpr >> 5;   // warps per row
  if ((int)threadIdx.x < n) {   // thread r decides row r
    const int r = threadIdx.x;
    float a = 0.f, b = 0.f, c = 0.f, m = 0.f, pn = 0.f, pd = 0.f;
    for (int w = r * wpr; w < (r + 1) * wpr; ++w) {
      a += s_red[w][0];
      b += s_red[w][1];
      c += s_red[w][2];
      m += s_red[w][3];
      pn += s_red[w][4];
      pd += s_red[w][5];
    }
    s_mu[r] = smode == NORM_LN ? m / D : 0.f;
    const int tok = tok_r;
    int ex = 0;
    if (test) {
      const float cs = exit_similarity(metric, a, b, c, pn, pd);
      if (sim) sim[(size_t)tok * n_layers + (layer - 1)] = cs;
      const int f = forced_r;
      if (f != 0 && (f < 2 || f > n_layers)) atomicOr(err, ERRW_FORCED);
      ex = (f > 0) ? (f == layer) : (cs >= delta);
    }
    s_dst[r] = ex;
    s_tok[r] = tok;
    s_w[r] = a > 0.f ? rsqrtf(a) : 0.f;
  }
  __syncthreads();
  if (threadIdx.x == 0) {   // stable compaction (n <= 16)
    int e = 0, k = 0;
    for (int r = 0; r < n; ++r) {
      const int tok = s_tok[r];
      // all-at-once: the decision of the sequence's last prompt token (a later row)
      const int rl = aao_len ? min(n - 1, r + (aao_len - 1 - tok_pos[tok])) : r;
      if (s_dst[rl]) {
        s_dst[r] = -1 - (base + e);
        exit_tok[base + e] = tok;
        if (exit_layer_out) exit_layer_out[tok] = layer;
        ++e;
      } else {
        s_dst[r] = k;
        row_tok_next[k] = tok;
        ++k;
      }
    }
    ctr[CTR_ACTIVE + (par ^ 1)] = k;
    ctr[CTR_EXITED] = base + e;
    ctr[CTR_PREFIX + layer] = base + e;
  }
  __syncthreads();
  if (xhat_next) {
    // the kept rows standardised for the next layer's attention input, as the
    // standardisation kernel computes them (two-pass: the centred second moment from the
    // registers); written to row d0 of xhat_next in bf16
    const float mu = row < n ? s_mu[row] : 0.f;
    float c2 = 0.f;
    if (row < n) {
#pragma unroll
      for (int j = 0; j < V; ++j)
        if (sub + j * tpr < D4) {
          const float4 a = xs[j];
          c2 += (a.x - mu) * (a.x - mu) + (a.y - mu) * (a.y - mu) + (a.z - mu) * (a.z - mu) + (a.w - mu) * (a.w - mu);
        }
    }
    c2 = warp_sum(c2);
    if (lane == 0) s_red[warp][0] = c2;
    __syncthreads();
    if (row < n && s_dst[row] >= 0) {
      float t = 0.f;
      for (int w = row * wpr; w < (row + 1) * wpr; ++w) t += s_red[w][0];
      const float rs = smode == NORM_COPY ? 1.f : rsqrtf(t / D + seps);
      const float m0 = smode == NORM_COPY ? 0.f : mu;
      uint2* o = reinterpret_cast<uint2*>(xhat_next + (size_t)s_dst[row] * D);
#pragma unroll
      for (int j = 0; j < V; ++j) {
        const int v = sub + j * tpr;
        if (v < D4) {
          const float4 a = xs[j];
          const __nv_bfloat162 lo = __floats2bfloat162_rn((a.x - m0) * rs, (a.y - m0) * rs);
          const __nv_bfloat162 hi = __floats2bfloat162_rn((a.z - m0) * rs, (a.w - m0) * rs);
          uint2 u;
          u.x = *reinterpret_cast<const uint32_t*>(&lo);
          u.y = *reinterpret_cast<const uint32_t*>(&hi);
          o[v] = u;
        }
      }
    }
  }
  if (row >= n) return;
  const int d0 = s_dst[row];
  if (d0 >= 0) {
    const float w = s_w[row];
    float4* xn = reinterpret_cast<float4*>(Xnext + (size_t)d0 * D);
    float4* inn = reinterpret_cast<float4*>(Inext + (size_t)d0 * D);
#pragma unroll
    for (int j = 0; j < V; ++j) {
      const int v = sub + j * tpr;
      if (v < D4) {
        const float4 a = xs[j], c = xi[j];
        xn[v] = a;
        inn[v] = make_float4(c.x + a.x * w, c.y + a.y * w, c.z + a.z * w, c.w + a.w * w);
      }
    }
  } else {
    const size_t kk = (size_t)(-1 - d0);
    float4* hs = reinterpret_cast<float4*>(hsm_s + kk * D);
    float4* hp = reinterpret_cast<float4*>(hsm_prev + kk * D);
    float4* hi = reinterpret_cast<float4*>(hsm_I + kk * D);
#pragma unroll
    for (int j = 0; j < V; ++j) {
      const int v = sub + j * tpr;
      if (v < D4) {
        hs[v] = xs[j];
        hp[v] = xp[j];
        hi[v] = xi[j];
      }
    }
  }
}

bool launch_exit_small(cudaStream_t st, const float* Xin, const float* Xout, const float* I, int first, int D,
                       int* ctr, int par, const int* row_tok, int* row_tok_next, const int* forced, int layer,
                       int n_layers, const float* delta_p, int test, float* sim, int* exit_tok, int* exit_layer_out,
                       float* Xnext, float* Inext, float* hsm_s, float* hsm_prev, float* hsm_I, int max_rows,
                       bf16* xhat_next, int smode, float seps, int metric, int aao_len, const int* tok_pos,
                       unsigned* err) {
  int rshift = 0;
  while ((1 << rshift) < max_rows) ++rshift;
  const bool aligned = ((uintptr_t)Xin | (uintptr_t)Xout | (uintptr_t)I | (uintptr_t)Xnext | (uintptr_t)Inext |
                        (uintptr_t)hsm_s | (uintptr_t)hsm_prev | (uintptr_t)hsm_I) % 16 == 0;
  if (max_rows <= 16 && D % 4 == 0 && D / 4 <= EXD_V * (EXD_THREADS >> rshift) && aligned) {
    auto* kern = D / 4 <= 2 * (EXD_THREADS >> rshift) ? exit_decode_kernel<2> : exit_decode_kernel<EXD_V>;
    launch_k(kern, 1, EXD_THREADS, 0, st, Xin, Xout, I, first, D, ctr, par, row_tok, row_tok_next, forced,
             layer, n_layers, delta_p, test, sim, exit_tok, exit_layer_out, Xnext, Inext, hsm_s, hsm_prev, hsm_I,
             rshift, max_rows, xhat_next, smode, seps, metric, aao_len, tok_pos, err);
    return true;
  }
  launch_k(exit_small_kernel, 1, 256, 0, st, Xin, Xout, I, first, D, ctr, par, row_tok, row_tok_next, forced, layer,
           n_layers, delta_p, test, sim, exit_tok, exit_layer_out, Xnext, Inext, hsm_s, hsm_prev, hsm_I, metric,
           aao_len, tok_pos, err);
  return false;
}

__global__ void set_float_kernel(float* p, float v) {
  PDL_ENTRY(); *p = v; }
void launch_set_float(cudaStream_t st, float* p, float v) { launch_k(set_float_kernel, 1, 1, 0, st, p, v); }

// Span timer: every used launch site's span into its class total; the site is reset.
__global__ void span_collect_kernel(SpanSite* sites, int n, SpanTotal* tot, int n_cls) {
  PDL_ENTRY();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    SpanSite& s = sites[i];
    const unsigned long long t0 = s.t0, t1 = s.t1;
    if (t0 == ~0ull) continue;
    if (t1 > t0 && s.cls >= 0 && s.cls < n_cls) {
      atomicAdd(&tot[s.cls].ns, t1 - t0);
      atomicAdd(&tot[s.cls].n, 1ull);
    }
    s.t0 = ~0ull;
    s.t1 = 0ull;
  }
}

void launch_span_collect(cudaStream_t st, SpanSite* sites, int n, SpanTotal* tot, int n_cls) {
  launch_k(span_collect_kernel, 1, 1024, 0, st, sites, n, tot, n_cls);
}

// Generation-step staging: the caller's inputs into the library's fixed buffers (the captured
// step reads only those), in one launch instead of a kernel and two copies.
__global__ void stage_in_kernel(float* d_delta, float delta, const int* tokens, int* dec_tok, const int* forced,
                                int* dec_forced, int batch) {
  PDL_ENTRY();
  if (threadIdx.x == 0) *d_delta = delta;
  for (int b = threadIdx.x; b < batch; b += blockDim.x) {
    dec_tok[b] = tokens[b];
    dec_forced[b] = forced ? forced[b] : 0;
  }
}
void launch_stage_in(cudaStream_t st, float* d_delta, float delta, const int* tokens, int* dec_tok, const int* forced,
                     int* dec_forced, int batch) {
  launch_k(stage_in_kernel, 1, 32, 0, st, d_delta, delta, tokens, dec_tok, forced, dec_forced, batch);
}

// ... and the step's outputs out of them into the caller's buffers (each optional).
__global__ void stage_out_kernel(int batch, const int* dec_exit, int* exit_out, const int* dec_next, int* next_out,
                                 const float* logits, float* logits_out, long long n_logits, const float* sim,
                                 float* sim_out, int n_sim) {
  PDL_ENTRY();
  const long long i0 = (long long)blockIdx.x * blockDim.x + threadIdx.x, step = (long long)gridDim.x * blockDim.x;
  for (long long i = i0; i < batch; i += step) {
    if (exit_out) exit_out[i] = dec_exit[i];
    if (next_out) next_out[i] = dec_next[i];
  }
  if (sim_out)
    for (long long i = i0; i < n_sim; i += step) sim_out[i] = sim[i];
  if (logits_out)
    for (long long i = i0; i < n_logits; i += step) logits_out[i] = logits[i];
}
void launch_stage_out(cudaStream_t st, int batch, const int* dec_exit, int* exit_out, const int* dec_next,
                      int* next_out, const float* logits, float* logits_out, long long n_logits, const float* sim,
                      float* sim_out, int n_sim) {
  const int grid = logits_out ? (int)std::min<long long>(304, (n_logits + 255) / 256) : 1;
  launch_k(stage_out_kernel, std::max(grid, 1), 256, 0, st, batch, dec_exit, exit_out, dec_next, next_out, logits,
           logits_out, n_logits, sim, sim_out, n_sim);
}

// After layer N: the remaining active rows' s_N are their final states.
__global__ void final_scatter_kernel(const float* X, int D, const int* n_rows, const int* row_tok, float* final_,
                                     int* exit_layer_out, int n_layers) {
  PDL_ENTRY();
  const int r = blockIdx.x;
  if (r >= *n_rows) return;
  const int tok = row_tok[r];
  for (int d = threadIdx.x; d < D; d += blockDim.x) final_[(size_t)tok * D + d] = X[(size_t)r * D + d];
  if (threadIdx.x == 0 && exit_layer_out) exit_layer_out[tok] = n_layers;
}

// final_scatter_kernel that also writes the row standardised for the output head (hmode
// NORM_RMS / NORM_LN, the head's gain and shift folded into its weights) at the token's head
// row of xhead (generation steps: token = sequence); the row is held in registers.
template <int EPT>
__global__ void __launch_bounds__(1024) final_scatter_head_kernel(const float* X, int D, const int* n_rows,
                                                                  const int* row_tok, float* final_,
                                                                  int* exit_layer_out, int n_layers, bf16* xhead,
                                                                  int hmode, float heps);


// ---------------------------------------------------------------------------
// Hidden State Mapper, non-GEMM steps (Sec. 4.2, App. B Table S1)
// ---------------------------------------------------------------------------
// Hidden State Mapper row steps (Table S1).  One CTA per row.  The register-resident
// kernels hold a row as EPT elements per thread (d = threadIdx.x + j * blockDim.x), issue
// every load of the row before the first reduction and compute from registers, so a row
// costs one round of memory latency instead of one per strided loop iteration (these
// kernels run on a handful of rows in a generation step, where latency is the cost).  Longer
// rows (above 4096 elements for the convolution step, 8192 for the others) take the
// strided-loop kernels further below.
// ---------------------------------------------------------------------------

template <int EPT>
__device__ __forceinline__ void hsm_load_row(const float* __restrict__ p, int n, float (&v)[EPT]) {
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    v[j] = d < n ? p[d] : 0.f;
  }
}

// Block-wide sums of NV values in a fixed order (blockDim.x a multiple of 32); red holds
// 32 * NV floats.  Every thread gets the sums.
template <int NV>
__device__ __forceinline__ void block_sum_n(float (&v)[NV], float* red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = warp_sum(v[i]);
  __syncthreads();
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < NV; ++i) red[w * NV + i] = v[i];
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    float t = 0.f;
    for (int k = 0; k < nw; ++k) t += red[k * NV + i];
    v[i] = t;
  }
}

// embed_kernel with the row held in registers (EPT elements per thread, all loads issued
// before the first reduction): rows of up to 16 x blockDim.x elements.
template <typename T, int EPT>
__global__ void __launch_bounds__(256) embed_reg_kernel(const int* tokens, int n_tok, const int* tok_pos, const T* E,
                                                        const T* P, const float* type_emb, const float* g,
                                                        const float* b, int family, int D, int V, float eps, float* X,
                                                        unsigned* err, bf16* xhat, int smode, float seps) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int t = blockIdx.x;
  if (t >= n_tok) return;
  int tok = tokens[t];
  if (tok < 0 || tok >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERRW_TOKEN);
    tok = 0;
  }
  const int pos = tok_pos[t];
  float v[EPT];
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    float x = 0.f;
    if (d < D) {
      x = to_f(E[(size_t)tok * D + d]);
      if (P) x += to_f(P[(size_t)pos * D + d]);
      if (type_emb) x += type_emb[d];
    }
    v[j] = x;
  }
  float* x = X + (size_t)t * D;
  float s1[1] = {0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) s1[0] += v[j];
  const bool ln = family == 2 || smode == NORM_LN;
  if (family != 2) {
#pragma unroll
    for (int j = 0; j < EPT; ++j) {
      const int d = threadIdx.x + j * blockDim.x;
      if (d < D) x[d] = v[j];
    }
    if (!xhat) return;
  }
  float mu = 0.f;
  if (ln) {
    block_sum_n<1>(s1, red);
    mu = s1[0] / D;
  }
  float s2[1] = {0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    const float c = d < D ? v[j] - mu : 0.f;
    s2[0] += c * c;
  }
  block_sum_n<1>(s2, red);
  if (family != 2) {
    const float rs = smode == NORM_COPY ? 1.f : rsqrtf(s2[0] / D + seps);
    const float m0 = smode == NORM_COPY ? 0.f : mu;
#pragma unroll
    for (int j = 0; j < EPT; ++j) {
      const int d = threadIdx.x + j * blockDim.x;
      if (d < D) xhat[(size_t)t * D + d] = __float2bfloat16_rn((v[j] - m0) * rs);
    }
    return;
  }
  const float rstd = rsqrtf(s2[0] / D + eps);
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) x[d] = (v[j] - mu) * rstd * g[d] + b[d];
  }
}

// Three separately RMS-normalised rows (shared gain g0), then the 3x3 convolution with
// padding (0, 1): c0[t] = b + sum_a sum_u w[a][u] Xn_a[t + u - 1], Xn_a = x_a rstd_a g0.
// Dynamic shared memory: the three normalised rows, 3 * D floats.
template <typename T, int EPT>
__global__ void __launch_bounds__(256) hsm_prep_kernel(const float* hs, const float* hp, const float* hI, DevRange rows, int D,
                                const float* g0, const float* conv /* 9 taps + bias */, float eps, float* c0f,
                                T* c0t) {
  PDL_ENTRY();
  extern __shared__ float s_xn[];
  __shared__ float red[32 * 3];
  const int kb = rows.b(), ke = rows.e();
  for (int k = kb + blockIdx.x; k < ke; k += gridDim.x) {   // rows of the live range, in turn
  float xa[EPT], xb[EPT], xc[EPT], g[EPT];
  hsm_load_row(hs + (size_t)k * D, D, xa);
  hsm_load_row(hp + (size_t)k * D, D, xb);
  hsm_load_row(hI + (size_t)k * D, D, xc);
  hsm_load_row(g0, D, g);
  float w[10];
#pragma unroll
  for (int i = 0; i < 10; ++i) w[i] = conv[i];
  float ss[3] = {0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    ss[0] += xa[j] * xa[j];
    ss[1] += xb[j] * xb[j];
    ss[2] += xc[j] * xc[j];
  }
  block_sum_n<3>(ss, red);
  const float sa = rsqrtf(ss[0] / D + eps), sb = rsqrtf(ss[1] / D + eps), sc = rsqrtf(ss[2] / D + eps);
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) {
      s_xn[d] = xa[j] * sa * g[j];
      s_xn[D + d] = xb[j] * sb * g[j];
      s_xn[2 * D + d] = xc[j] * sc * g[j];
    }
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int t = threadIdx.x + j * blockDim.x;
    if (t >= D) continue;
    float acc = w[9];
#pragma unroll
    for (int a = 0; a < 3; ++a) {
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int tt = t + u - 1;
        if (tt >= 0 && tt < D) acc += w[a * 3 + u] * s_xn[a * D + tt];
      }
    }
    c0f[(size_t)k * D + t] = acc;
    c0t[(size_t)k * D + t] = from_f<T>(acc);
  }
  }
}

// h4 = RMSNorm_g1(h3) + h1 (the MLP's addition), rounded for FC4.
template <typename T, int EPT>
__global__ void __launch_bounds__(1024) hsm_mid_kernel(const float* h3, const float* h1, DevRange rows, int m1, const float* g1, float eps,
                               T* h4) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int kb = rows.b(), ke = rows.e();
  for (int k = kb + blockIdx.x; k < ke; k += gridDim.x) {
  float a[EPT], b[EPT];
  hsm_load_row(h3 + (size_t)k * m1, m1, a);
  hsm_load_row(h1 + (size_t)k * m1, m1, b);
  float s2[1] = {0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) s2[0] += a[j] * a[j];
  block_sum_n<1>(s2, red);
  const float sc = rsqrtf(s2[0] / m1 + eps);
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < m1) h4[(size_t)k * m1 + d] = from_f<T>(a[j] * sc * g1[d] + b[j]);
  }
  }
}

// s~ = RMSNorm_g2(h5) + c0 (the final addition); written to the token's final state,
// and standardised (the attention-input normalisation of the family) for the fills.
// identity != 0: s~ = s_i* (test switch replacing the HSM).
// xhead (optional, generation steps): the same standardised row also at the token's head row.
template <typename T, int EPT>
__global__ void __launch_bounds__(1024) hsm_out_kernel(const float* h5, const float* c0f, const float* hs, int identity, DevRange rows, int D,
                               const float* g2, float eps, const int* exit_tok, float* final_, T* xfill,
                               int fill_mode, float norm_eps, T* xhead) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int kb = rows.b(), ke = rows.e();
  for (int k = kb + blockIdx.x; k < ke; k += gridDim.x) {
  const int tok = exit_tok[k];
  float f[EPT];
  if (identity) {
    hsm_load_row(hs + (size_t)k * D, D, f);
  } else {
    float c[EPT];
    hsm_load_row(h5 + (size_t)k * D, D, f);
    hsm_load_row(c0f + (size_t)k * D, D, c);
    float s2[1] = {0.f};
#pragma unroll
    for (int j = 0; j < EPT; ++j) s2[0] += f[j] * f[j];
    block_sum_n<1>(s2, red);
    const float sc = rsqrtf(s2[0] / D + eps);
#pragma unroll
    for (int j = 0; j < EPT; ++j) {
      const int d = threadIdx.x + j * blockDim.x;
      f[j] = d < D ? f[j] * sc * g2[d] + c[j] : 0.f;
    }
  }
  float* fo = final_ + (size_t)tok * D;
  T* o = xfill + (size_t)k * D;
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) fo[d] = f[j];
  }
  if (fill_mode == NORM_COPY) {
#pragma unroll
    for (int j = 0; j < EPT; ++j) {
      const int d = threadIdx.x + j * blockDim.x;
      if (d < D) o[d] = from_f<T>(f[j]);
    }
    continue;
  }
  float mu = 0.f;
  if (fill_mode == NORM_LN) {
    float s[1] = {0.f};
#pragma unroll
    for (int j = 0; j < EPT; ++j) s[0] += f[j];
    block_sum_n<1>(s, red);
    mu = s[0] / D;
  }
  float v[1] = {0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    const float c = d < D ? f[j] - mu : 0.f;
    v[0] += c * c;
  }
  block_sum_n<1>(v, red);
  const float rstd = rsqrtf(v[0] / D + norm_eps);
  T* oh = xhead ? xhead + (size_t)tok * D : nullptr;
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) {
      const T x = from_f<T>((f[j] - mu) * rstd);
      o[d] = x;
      if (oh) oh[d] = x;
    }
  }
  }
}

template <int EPT>
__global__ void __launch_bounds__(1024) final_scatter_head_kernel(const float* X, int D, const int* n_rows,
                                                                  const int* row_tok, float* final_,
                                                                  int* exit_layer_out, int n_layers, bf16* xhead,
                                                                  int hmode, float heps) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int r = blockIdx.x;
  if (r >= *n_rows) return;
  const int tok = row_tok[r];
  float f[EPT];
  hsm_load_row(X + (size_t)r * D, D, f);
  float* fo = final_ + (size_t)tok * D;
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) fo[d] = f[j];
  }
  if (threadIdx.x == 0 && exit_layer_out) exit_layer_out[tok] = n_layers;
  float mu = 0.f;
  if (hmode == NORM_LN) {
    float s[1] = {0.f};
#pragma unroll
    for (int j = 0; j < EPT; ++j) s[0] += f[j];
    block_sum_n<1>(s, red);
    mu = s[0] / D;
  }
  float v[1] = {0.f};
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    const float c = d < D ? f[j] - mu : 0.f;
    v[0] += c * c;
  }
  block_sum_n<1>(v, red);
  const float rstd = rsqrtf(v[0] / D + heps);
  bf16* oh = xhead + (size_t)tok * D;
#pragma unroll
  for (int j = 0; j < EPT; ++j) {
    const int d = threadIdx.x + j * blockDim.x;
    if (d < D) oh[d] = __float2bfloat16_rn((f[j] - mu) * rstd);
  }
}

// Strided-loop forms of the three kernels above, for the longer rows.
// Three separately RMS-normalised rows (shared gain g0), then the 3x3 convolution with
// padding (0, 1): c0[t] = b + sum_a sum_u w[a][u] x_a[t + u - 1].
template <typename T>
__global__ void hsm_prep_loop_kernel(const float* hs, const float* hp, const float* hI, DevRange rows, int D,
                                const float* g0, const float* conv /* 9 taps + bias */, float eps, float* c0f,
                                T* c0t) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int k = rows.b() + blockIdx.x;
  if (k >= rows.e()) return;
  const float* x[3] = {hs + (size_t)k * D, hp + (size_t)k * D, hI + (size_t)k * D};
  float sc[3];
#pragma unroll
  for (int a = 0; a < 3; ++a) {
    float s2 = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s2 += x[a][d] * x[a][d];
    sc[a] = rsqrtf(block_sum(s2, red) / D + eps);
  }
  for (int t = threadIdx.x; t < D; t += blockDim.x) {
    float acc = conv[9];
#pragma unroll
    for (int a = 0; a < 3; ++a) {
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int tt = t + u - 1;
        if (tt >= 0 && tt < D) acc += conv[a * 3 + u] * (x[a][tt] * sc[a] * g0[tt]);
      }
    }
    c0f[(size_t)k * D + t] = acc;
    c0t[(size_t)k * D + t] = from_f<T>(acc);
  }
}

// h4 = RMSNorm_g1(h3) + h1 (the MLP's addition), rounded for FC4.
template <typename T>
__global__ void hsm_mid_loop_kernel(const float* h3, const float* h1, DevRange rows, int m1, const float* g1, float eps,
                               T* h4) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int k = rows.b() + blockIdx.x;
  if (k >= rows.e()) return;
  const float* a = h3 + (size_t)k * m1;
  float s2 = 0.f;
  for (int d = threadIdx.x; d < m1; d += blockDim.x) s2 += a[d] * a[d];
  const float sc = rsqrtf(block_sum(s2, red) / m1 + eps);
  for (int d = threadIdx.x; d < m1; d += blockDim.x)
    h4[(size_t)k * m1 + d] = from_f<T>(a[d] * sc * g1[d] + h1[(size_t)k * m1 + d]);
}

// s~ = RMSNorm_g2(h5) + c0 (the final addition); written to the token's final state,
// and standardised (the attention-input normalisation of the family) for the fills.
// identity != 0: s~ = s_i* (test switch replacing the HSM).
template <typename T>
__global__ void hsm_out_loop_kernel(const float* h5, const float* c0f, const float* hs, int identity, DevRange rows, int D,
                               const float* g2, float eps, const int* exit_tok, float* final_, T* xfill,
                               int fill_mode, float norm_eps, T* xhead) {
  PDL_ENTRY();
  __shared__ float red[32];
  const int k = rows.b() + blockIdx.x;
  if (k >= rows.e()) return;
  const int tok = exit_tok[k];
  float* f = final_ + (size_t)tok * D;
  if (identity) {
    for (int d = threadIdx.x; d < D; d += blockDim.x) f[d] = hs[(size_t)k * D + d];
  } else {
    const float* a = h5 + (size_t)k * D;
    float s2 = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s2 += a[d] * a[d];
    const float sc = rsqrtf(block_sum(s2, red) / D + eps);
    for (int d = threadIdx.x; d < D; d += blockDim.x) f[d] = a[d] * sc * g2[d] + c0f[(size_t)k * D + d];
  }
  __syncthreads();
  T* o = xfill + (size_t)k * D;
  if (fill_mode == NORM_COPY) {
    for (int d = threadIdx.x; d < D; d += blockDim.x) o[d] = from_f<T>(f[d]);
    return;
  }
  float mu = 0.f;
  if (fill_mode == NORM_LN) {
    float s = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s += f[d];
    mu = block_sum(s, red) / D;
  }
  float s2 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float c = f[d] - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(block_sum(s2, red) / D + norm_eps);
  T* oh = xhead ? xhead + (size_t)tok * D : nullptr;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const T x = from_f<T>((f[d] - mu) * rstd);
    o[d] = x;
    if (oh) oh[d] = x;
  }
}

// ---------------------------------------------------------------------------
// greedy token: argmax with the lowest index on ties
// ---------------------------------------------------------------------------
__global__ void argmax_kernel(const float* logits, int V, int rows, int* out) {
  PDL_ENTRY();
  __shared__ float sv[32];
  __shared__ int si[32];
  const int r = blockIdx.x;
  if (r >= rows) return;
  const float* l = logits + (size_t)r * V;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int v = threadIdx.x; v < V; v += blockDim.x) {
    const float x = l[v];
    if (x > bv || (x == bv && v < bi)) {
      bv = x;
      bi = v;
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > bv || (ov == bv && oi < bi)) {
      bv = ov;
      bi = oi;
    }
  }
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) {
    sv[w] = bv;
    si[w] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int k = 1; k < (int)(blockDim.x >> 5); ++k)
      if (sv[k] > bv || (sv[k] == bv && si[k] < bi)) {
        bv = sv[k];
        bi = si[k];
      }
    out[r] = bi == 0x7fffffff ? 0 : bi;
  }
}

// Rows of the last position of each sequence (decoder head) or of position 0 (encoder).
__global__ void head_rows_kernel(int batch, int prompt_len, int last, int* rows) {
  PDL_ENTRY();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < batch) rows[b] = b * prompt_len + (last ? prompt_len - 1 : 0);
}

// ---------------------------------------------------------------------------
// skipped-layer fill input: bucket tokens by exit layer (ascending) so that the rows of
// skipped layer r (tokens with i* < r) are a prefix, and standardise s~ once.
// ---------------------------------------------------------------------------
// The histogram and the scan in one CTA (histogram in shared memory): one launch instead of
// a memset and two kernels ahead of the scatter.  Calls of at most FILL_PLAN_ROWS tokens
// (generation steps, small fills) also place and standardise the rows here, one warp per row,
// so that the whole pre-pass is this one launch.
constexpr int FILL_PLAN_ROWS = 32;
// One row standardised (the attention-input normalisation of the family) by one warp.
template <typename T>
__device__ __forceinline__ void plan_row(const T* x, T* o, int D, int mode, float eps, int lane) {
  constexpr int E = 16 / sizeof(T);   // elements per 16-byte piece
  const int nch = D / (32 * E);       // pieces per lane
  if (D % (32 * E) == 0 && nch <= 16 && (((uintptr_t)x | (uintptr_t)o) & 15) == 0) {
    // the row in registers, every load issued before the first reduction (one memory round
    // trip instead of one per strided loop iteration)
    uint4 r[16];
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < nch) r[i] = reinterpret_cast<const uint4*>(x)[lane + 32 * i];
    auto val = [&](int i, int e) { return to_f(reinterpret_cast<const T*>(&r[i])[e]); };
    float mu = 0.f, s2 = 0.f;
    if (mode == NORM_LN) {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (i < nch)
#pragma unroll
          for (int e = 0; e < E; ++e) mu += val(i, e);
      mu = warp_sum(mu) / D;
    }
    float rstd = 1.f;
    if (mode != NORM_COPY) {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (i < nch)
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const float c = val(i, e) - mu;
            s2 += c * c;
          }
      rstd = rsqrtf(warp_sum(s2) / D + eps);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < nch) {
        uint4 w;
        T* wt = reinterpret_cast<T*>(&w);
#pragma unroll
        for (int e = 0; e < E; ++e) wt[e] = mode == NORM_COPY ? reinterpret_cast<const T*>(&r[i])[e]
                                                             : from_f<T>((val(i, e) - mu) * rstd);
        reinterpret_cast<uint4*>(o)[lane + 32 * i] = w;
      }
    return;
  }
  if (mode == NORM_COPY) {
    for (int d = lane; d < D; d += 32) o[d] = x[d];
    return;
  }
  float mu = 0.f;
  if (mode == NORM_LN) {
    float sm = 0.f;
    for (int d = lane; d < D; d += 32) sm += to_f(x[d]);
    mu = warp_sum(sm) / D;
  }
  float s2 = 0.f;
  for (int d = lane; d < D; d += 32) {
    const float c = to_f(x[d]) - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(warp_sum(s2) / D + eps);
  for (int d = lane; d < D; d += 32) o[d] = from_f<T>((to_f(x[d]) - mu) * rstd);
}

template <typename T>
__global__ void __launch_bounds__(512) fill_plan_kernel(const T* h, int D, const int* exit_layer, int n, int n_layers,
                                                         int* hist, int* start, int* cursor, int* sorted_tok, T* xs,
                                                         int mode, float eps, unsigned* err) {
  PDL_ENTRY();
  extern __shared__ int s_hist[];   // [n_layers + 2] counts, then [n_layers + 2] running slots
  int* s_cur = s_hist + n_layers + 2;
  __shared__ int s_slot[FILL_PLAN_ROWS];
  for (int l = threadIdx.x; l < n_layers + 2; l += blockDim.x) s_hist[l] = 0;
  __syncthreads();
  bool bad = false;
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    int l = exit_layer[j];
    if (l < 1 || l > n_layers) {
      bad = true;
      l = n_layers;
    }
    atomicAdd(&s_hist[l], 1);
  }
  if (bad) atomicOr(err, ERRW_EXIT_LAYER);
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int l = 0; l <= n_layers + 1; ++l) {
      start[l] = acc;
      s_cur[l] = acc;
      cursor[l] = 0;
      hist[l] = s_hist[l];
      if (l >= 1 && l <= n_layers) acc += s_hist[l];
    }
  }
  if (n > FILL_PLAN_ROWS) return;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x < n) {
    int l = exit_layer[threadIdx.x];
    if (l < 1 || l > n_layers) l = n_layers;
    const int slot = atomicAdd(&s_cur[l], 1);
    s_slot[threadIdx.x] = slot;
    sorted_tok[slot] = threadIdx.x;
  }
  __syncthreads();
  for (int row = warp; row < n; row += blockDim.x >> 5)
    plan_row(h + (size_t)row * D, xs + (size_t)s_slot[row] * D, D, mode, eps, lane);
}

template <typename T>
__global__ void fill_scatter_kernel(const T* h, int n, int D, const int* exit_layer, int n_layers, const int* start,
                                    int* cursor, int* sorted_tok, T* xs, int mode, float eps) {
  PDL_ENTRY();
  __shared__ float red[32];
  __shared__ int s_slot;
  const int j = blockIdx.x;
  if (j >= n) return;
  if (threadIdx.x == 0) {
    int l = exit_layer[j];
    if (l < 1 || l > n_layers) l = n_layers;
    s_slot = start[l] + atomicAdd(&cursor[l], 1);
    sorted_tok[s_slot] = j;
  }
  __syncthreads();
  const int slot = s_slot;
  const T* x = h + (size_t)j * D;
  T* o = xs + (size_t)slot * D;
  if (mode == NORM_COPY) {
    for (int d = threadIdx.x; d < D; d += blockDim.x) o[d] = x[d];
    return;
  }
  float mu = 0.f;
  if (mode == NORM_LN) {
    float s = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) s += to_f(x[d]);
    mu = block_sum(s, red) / D;
  }
  float s2 = 0.f;
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    const float c = to_f(x[d]) - mu;
    s2 += c * c;
  }
  const float rstd = rsqrtf(block_sum(s2, red) / D + eps);
  for (int d = threadIdx.x; d < D; d += blockDim.x) o[d] = from_f<T>((to_f(x[d]) - mu) * rstd);
}

// ---------------------------------------------------------------------------
// load-time repacking: W'[n, k] = W[src(n), k] * gamma[k] (rounded once),
// b'[n] = b[src(n)] + sum_k W[src(n), k] * beta[k]
// ---------------------------------------------------------------------------
template <typename T>
__global__ void fold_rows_kernel(T* dst, int ld_dst, const T* src, int n_rows, int K, const float* gamma,
                                 const float* beta, const float* bias_in, float* bias_out, int row_mode) {
  PDL_ENTRY();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= n_rows) return;
  const int n = warp;
  // row_mode 0: dst row = n.  1 / 2: gate / up of a SwiGLU pair, interleaved in blocks of 16.
  // row_mode >= 8: rotary head of row_mode features -- the rotate-half pair (i, i + hd/2)
  // lands on adjacent rows (2i, 2i + 1).
  int drow = n;
  if (row_mode == 1) drow = (n / 16) * 32 + (n % 16);
  if (row_mode == 2) drow = (n / 16) * 32 + 16 + (n % 16);
  if (row_mode >= 8) {
    const int hd = row_mode, half = hd / 2, h = n / hd, i = n % hd;
    drow = h * hd + (i < half ? 2 * i : 2 * (i - half) + 1);
  }
  const T* s = src + (size_t)n * K;
  T* o = dst + (size_t)drow * ld_dst;
  float acc = 0.f;
  for (int k = lane; k < K; k += 32) {
    const float w = to_f(s[k]);
    o[k] = gamma ? from_f<T>(w * gamma[k]) : s[k];
    if (beta) acc += w * beta[k];
  }
  acc = warp_sum(acc);
  if (lane == 0 && bias_out) bias_out[drow] = (bias_in ? bias_in[n] : 0.f) + acc;
}

template <typename T>
__global__ void to_f32_kernel(const T* src, float* dst, int n) {
  PDL_ENTRY();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) dst[i] = to_f(src[i]);
}

// Copy n_pos positions of one sequence / layer out of the paged cache.
template <typename T>
__global__ void read_kv_kernel(KVCacheView c, int layer0, int seq, int pos0, int n_pos, T* ko, T* vo) {
  PDL_ENTRY();
  const int p = blockIdx.x;
  if (p >= n_pos) return;
  const int per = c.n_kv_heads * c.head_dim;
  for (int e = threadIdx.x; e < per; e += blockDim.x) {
    const int h = e / c.head_dim, d = e % c.head_dim;
    const size_t off = c.offset(layer0, seq, pos0 + p, h) + d;
    ko[(size_t)p * per + e] = ((const T*)c.k)[off];
    vo[(size_t)p * per + e] = ((const T*)c.v)[off];
  }
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
void launch_pass_init(cudaStream_t st, int n_tok, int prompt_len, int decode, int* tok_seq, int* tok_pos,
                      int* row_tok, int* seq_len, int seq_cap, int max_pos, unsigned* err, int* ctr, int n_ctr,
                      float* sim, int n_layers, int* tok_exit) {
  launch_k(pass_init_kernel, cdiv(std::max(n_tok, n_ctr), 256), 256, 0, st, n_tok, prompt_len, decode, tok_seq, tok_pos,
           row_tok, seq_len, seq_cap, max_pos, err, ctr, n_ctr, sim, n_layers, tok_exit);
}

void launch_embed(cudaStream_t st, int dt, const int* tokens, int n_tok, const int* tok_pos, const void* E,
                  const void* P, const float* type_emb, const float* g, const float* b, int family, int D, int V,
                  float eps, float* X, unsigned* err, bf16* xhat, int smode, float seps) {
  if (D <= 16 * 256) {
#define EMB(T, EPT)                                                                                                  \
  launch_k(embed_reg_kernel<T, EPT>, n_tok, 256, 0, st, tokens, n_tok, tok_pos, (const T*)E, (const T*)P, type_emb, g, \
           b, family, D, V, eps, X, err, xhat, smode, seps)
    if (dt == 1) {
      if (D <= 4 * 256) EMB(bf16, 4);
      else EMB(bf16, 16);
    } else {
      if (D <= 4 * 256) EMB(float, 4);
      else EMB(float, 16);
    }
#undef EMB
    return;
  }
  if (dt == 1)
    launch_k(embed_kernel<bf16>, n_tok, 256, 0, st, tokens, n_tok, tok_pos, (const bf16*)E, (const bf16*)P, type_emb, g,
             b, family, D, V, eps, X, err, xhat, smode, seps);
  else
    launch_k(embed_kernel<float>, n_tok, 256, 0, st, tokens, n_tok, tok_pos, (const float*)E, (const float*)P, type_emb,
             g, b, family, D, V, eps, X, err, xhat, smode, seps);
}

void launch_standardize(cudaStream_t st, int dt, const float* X, int ldx, const int* in_rows, DevRange rows,
                        int max_rows, int D, int mode, float eps, void* out, int ld_out) {
  if (max_rows <= 0) return;
  if (dt == 1)
    launch_k(standardize_kernel<bf16>, row_grid(max_rows, 8), 256, 0, st, X, ldx, in_rows, rows, D, mode, eps, (bf16*)out, ld_out);
  else
    launch_k(standardize_kernel<float>, row_grid(max_rows, 8), 256, 0, st, X, ldx, in_rows, rows, D, mode, eps, (float*)out, ld_out);
}

void launch_layernorm_inplace(cudaStream_t st, float* X, DevRange rows, int max_rows, int D, const float* g,
                              const float* b, float eps) {
  if (max_rows <= 0) return;
  launch_k(layernorm_inplace_kernel, max_rows, 256, 0, st, X, rows, D, g, b, eps);
}

void launch_exit_decide(cudaStream_t st, const float* Xout, const float* I, const float* Xin, int D, DevRange rows,
                        int max_rows, const int* row_tok, const int* forced, int layer, int n_layers,
                        const float* delta_p, int test, int metric, float* sim, int* flag, float* inv_norm,
                        unsigned* err) {
  if (max_rows <= 0) return;
  launch_k(exit_decide_kernel, cdiv(max_rows, 8), 256, 0, st, Xout, I, Xin, D, rows, row_tok, forced, layer, n_layers,
           delta_p, test, metric, sim, flag, inv_norm, err);
}

void launch_exit_scan(cudaStream_t st, int* ctr, int in_parity, const int* flag, const int* row_tok,
                      int* row_tok_next, int* exit_tok, int* dst, int* exit_layer_out, int layer, int aao_len,
                      const int* tok_pos) {
  launch_k(exit_scan_kernel, 1, 1024, 0, st, ctr, in_parity, flag, row_tok, row_tok_next, exit_tok, dst, exit_layer_out,
           layer, aao_len, tok_pos);
}

void launch_exit_move(cudaStream_t st, const float* Xin, const float* Xout, const float* I, int first, int D,
                      const int* n_rows, int max_rows, const int* dst, const float* inv_norm, float* Xnext,
                      float* Inext, float* hsm_s, float* hsm_prev, float* hsm_I) {
  if (max_rows <= 0) return;
  launch_k(exit_move_kernel, row_grid(max_rows, 8), 256, 0, st, Xin, Xout, I, first, D, n_rows, dst, inv_norm, Xnext, Inext, hsm_s,
                                             hsm_prev, hsm_I);
}

void launch_final_scatter(cudaStream_t st, const float* X, int D, const int* n_rows, int max_rows, const int* row_tok,
                          float* final_, int* exit_layer_out, int n_layers) {
  if (max_rows <= 0) return;
  launch_k(final_scatter_kernel, max_rows, 256, 0, st, X, D, n_rows, row_tok, final_, exit_layer_out, n_layers);
}


// Threads per CTA of the register-resident mid / out kernels for a row of n elements (4
// elements per thread up to 1024, else 8), or 0 when the row needs the strided-loop kernel.
static int hsm_row_threads(int n) {
  if (n <= 4 * 256) return 256;
  if (n <= 8 * 512) return 512;
  if (n <= 8 * 1024) return 1024;
  return 0;
}

template <typename T, int EPT>
static void hsm_prep_go(cudaStream_t st, int thr, const float* hs, const float* hp, const float* hI, DevRange rows,
                        int max_rows, int D, const float* g0, const float* conv, float eps, float* c0f, void* c0t) {
  const size_t smem = (size_t)3 * D * sizeof(float);   // D <= 4096: at most 48 KB (+ static) -> opt in
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(hsm_prep_kernel<T, EPT>, cudaFuncAttributeMaxDynamicSharedMemorySize, 3 * 16 * 256 * 4);
    attr = true;
  }
  launch_k(hsm_prep_kernel<T, EPT>, hsm_grid(max_rows), thr, smem, st, hs, hp, hI, rows, D, g0, conv, eps, c0f,
           (T*)c0t);
}

void launch_hsm_prep(cudaStream_t st, int dt, const float* hs, const float* hp, const float* hI, DevRange rows,
                     int max_rows, int D, const float* g0, const float* conv, float eps, float* c0f, void* c0t) {
  if (max_rows <= 0) return;
  const int thr = D <= 16 * 256 ? 256 : 0;   // four row arrays in registers: 256 threads, 16 elements each
  if (thr == 0) {
    if (dt == 1)
      launch_k(hsm_prep_loop_kernel<bf16>, max_rows, 256, 0, st, hs, hp, hI, rows, D, g0, conv, eps, c0f, (bf16*)c0t);
    else
      launch_k(hsm_prep_loop_kernel<float>, max_rows, 256, 0, st, hs, hp, hI, rows, D, g0, conv, eps, c0f,
               (float*)c0t);
    return;
  }
  const bool small = D <= 4 * 256;
  if (dt == 1) {
    if (small) hsm_prep_go<bf16, 4>(st, thr, hs, hp, hI, rows, max_rows, D, g0, conv, eps, c0f, c0t);
    else hsm_prep_go<bf16, 16>(st, thr, hs, hp, hI, rows, max_rows, D, g0, conv, eps, c0f, c0t);
  } else {
    if (small) hsm_prep_go<float, 4>(st, thr, hs, hp, hI, rows, max_rows, D, g0, conv, eps, c0f, c0t);
    else hsm_prep_go<float, 16>(st, thr, hs, hp, hI, rows, max_rows, D, g0, conv, eps, c0f, c0t);
  }
}

void launch_hsm_mid(cudaStream_t st, int dt, const float* h3, const float* h1, DevRange rows, int max_rows, int m1,
                    const float* g1, float eps, void* h4) {
  if (max_rows <= 0) return;
  const int thr = hsm_row_threads(m1);
  if (thr == 0) {
    if (dt == 1) launch_k(hsm_mid_loop_kernel<bf16>, max_rows, 256, 0, st, h3, h1, rows, m1, g1, eps, (bf16*)h4);
    else launch_k(hsm_mid_loop_kernel<float>, max_rows, 256, 0, st, h3, h1, rows, m1, g1, eps, (float*)h4);
    return;
  }
  const bool small = m1 <= 4 * 256;
  if (dt == 1) {
    if (small) launch_k(hsm_mid_kernel<bf16, 4>, hsm_grid(max_rows), thr, 0, st, h3, h1, rows, m1, g1, eps, (bf16*)h4);
    else launch_k(hsm_mid_kernel<bf16, 8>, hsm_grid(max_rows), thr, 0, st, h3, h1, rows, m1, g1, eps, (bf16*)h4);
  } else {
    if (small) launch_k(hsm_mid_kernel<float, 4>, hsm_grid(max_rows), thr, 0, st, h3, h1, rows, m1, g1, eps, (float*)h4);
    else launch_k(hsm_mid_kernel<float, 8>, hsm_grid(max_rows), thr, 0, st, h3, h1, rows, m1, g1, eps, (float*)h4);
  }
}

void launch_hsm_out(cudaStream_t st, int dt, const float* h5, const float* c0f, const float* hs, int identity,
                    DevRange rows, int max_rows, int D, const float* g2, float eps, const int* exit_tok,
                    float* final_, void* xfill, int fill_mode, float norm_eps, void* xhead) {
  if (max_rows <= 0) return;
  const int thr = hsm_row_threads(D);
  if (thr == 0) {
    if (dt == 1)
      launch_k(hsm_out_loop_kernel<bf16>, max_rows, 256, 0, st, h5, c0f, hs, identity, rows, D, g2, eps, exit_tok,
               final_, (bf16*)xfill, fill_mode, norm_eps, (bf16*)xhead);
    else
      launch_k(hsm_out_loop_kernel<float>, max_rows, 256, 0, st, h5, c0f, hs, identity, rows, D, g2, eps, exit_tok,
               final_, (float*)xfill, fill_mode, norm_eps, (float*)xhead);
    return;
  }
  const bool small = D <= 4 * 256;
#define HSM_OUT(T, E)                                                                                              \
  launch_k(hsm_out_kernel<T, E>, hsm_grid(max_rows), thr, 0, st, h5, c0f, hs, identity, rows, D, g2, eps, exit_tok, final_, \
           (T*)xfill, fill_mode, norm_eps, (T*)xhead)
  if (dt == 1) {
    if (small) HSM_OUT(bf16, 4);
    else HSM_OUT(bf16, 8);
  } else {
    if (small) HSM_OUT(float, 4);
    else HSM_OUT(float, 8);
  }
#undef HSM_OUT
}

bool head_rows_supported(int D) { return hsm_row_threads(D) > 0; }

void launch_final_scatter_head(cudaStream_t st, const float* X, int D, const int* n_rows, int max_rows,
                               const int* row_tok, float* final_, int* exit_layer_out, int n_layers, bf16* xhead,
                               int hmode, float heps) {
  if (max_rows <= 0) return;
  const int thr = hsm_row_threads(D);
  if (D <= 4 * 256)
    launch_k(final_scatter_head_kernel<4>, max_rows, thr, 0, st, X, D, n_rows, row_tok, final_, exit_layer_out,
             n_layers, xhead, hmode, heps);
  else
    launch_k(final_scatter_head_kernel<8>, max_rows, thr, 0, st, X, D, n_rows, row_tok, final_, exit_layer_out,
             n_layers, xhead, hmode, heps);
}

// Two-stage argmax for long rows: ARGMAX_SPLIT blocks per row reduce slices to
// (value, index) pairs, one thread per row merges them (lowest index on ties).
constexpr int ARGMAX_SPLIT = 32;
__global__ void argmax_part_kernel(const float* logits, int V, int rows, float* pv, int* pi) {
  PDL_ENTRY();
  __shared__ float sv[32];
  __shared__ int si[32];
  const int r = blockIdx.x / ARGMAX_SPLIT, part = blockIdx.x % ARGMAX_SPLIT;
  if (r >= rows) return;
  const int chunk = (V + ARGMAX_SPLIT - 1) / ARGMAX_SPLIT;
  const int lo = part * chunk, hi = min(V, lo + chunk);
  const float* l = logits + (size_t)r * V;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  // the thread's values in groups of 8 loads in flight (ties: the lowest index wins in any order)
  for (int v0 = lo + threadIdx.x; v0 < hi; v0 += 8 * blockDim.x) {
    float x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int v = v0 + u * blockDim.x;
      x[u] = v < hi ? l[v] : -INFINITY;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int v = v0 + u * blockDim.x;
      if (v < hi && (x[u] > bv || (x[u] == bv && v < bi))) {
        bv = x[u];
        bi = v;
      }
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > bv || (ov == bv && oi < bi)) {
      bv = ov;
      bi = oi;
    }
  }
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) {
    sv[w] = bv;
    si[w] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int k = 1; k < (int)(blockDim.x >> 5); ++k)
      if (sv[k] > bv || (sv[k] == bv && si[k] < bi)) {
        bv = sv[k];
        bi = si[k];
      }
    pv[blockIdx.x] = bv;
    pi[blockIdx.x] = bi;
  }
}

__global__ void argmax_merge_kernel(const float* pv, const int* pi, int rows, int* out) {
  PDL_ENTRY();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= rows) return;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int k = 0; k < ARGMAX_SPLIT; ++k) {
    const float x = pv[r * ARGMAX_SPLIT + k];
    const int i = pi[r * ARGMAX_SPLIT + k];
    if (x > bv || (x == bv && i < bi)) {
      bv = x;
      bi = i;
    }
  }
  out[r] = bi == 0x7fffffff ? 0 : bi;
}

int launch_argmax(cudaStream_t st, const float* logits, int V, int rows, int* out, float* part_v, int* part_i) {
  if (rows <= 0) return 0;
  if (V <= 4096 || !part_v || !part_i) {
    launch_k(argmax_kernel, rows, 256, 0, st, logits, V, rows, out);
    return 1;
  }
  launch_k(argmax_part_kernel, rows * ARGMAX_SPLIT, 256, 0, st, logits, V, rows, part_v, part_i);
  launch_k(argmax_merge_kernel, cdiv(rows, 64), 64, 0, st, part_v, part_i, rows, out);
  return 2;
}

void launch_head_rows(cudaStream_t st, int batch, int prompt_len, int last, int* rows) {
  launch_k(head_rows_kernel, cdiv(batch, 128), 128, 0, st, batch, prompt_len, last, rows);
}

int launch_fill_sort(cudaStream_t st, int dt, const void* h, int n, int D, const int* exit_layer, int n_layers,
                     int* hist, int* start, int* cursor, int* sorted_tok, void* xs, int mode, float eps,
                     unsigned* err) {
  const size_t smem = (size_t)2 * (n_layers + 2) * sizeof(int);
  if (dt == 1)
    launch_k(fill_plan_kernel<bf16>, 1, 512, smem, st, (const bf16*)h, D, exit_layer, n, n_layers, hist, start, cursor,
             sorted_tok, (bf16*)xs, mode, eps, err);
  else
    launch_k(fill_plan_kernel<float>, 1, 512, smem, st, (const float*)h, D, exit_layer, n, n_layers, hist, start,
             cursor, sorted_tok, (float*)xs, mode, eps, err);
  if (n <= FILL_PLAN_ROWS) return 1;   // placed and standardised by the plan kernel
  if (dt == 1)
    launch_k(fill_scatter_kernel<bf16>, n, 256, 0, st, (const bf16*)h, n, D, exit_layer, n_layers, start, cursor,
                                                 sorted_tok, (bf16*)xs, mode, eps);
  else
    launch_k(fill_scatter_kernel<float>, n, 256, 0, st, (const float*)h, n, D, exit_layer, n_layers, start, cursor,
                                                  sorted_tok, (float*)xs, mode, eps);
  return 2;
}

void launch_fold_rows(cudaStream_t st, int dt, void* dst, int ld_dst, const void* src, int n_rows, int K,
                      const float* gamma, const float* beta, const float* bias_in, float* bias_out, int row_mode) {
  if (dt == 1)
    launch_k(fold_rows_kernel<bf16>, cdiv(n_rows, 8), 256, 0, st, (bf16*)dst, ld_dst, (const bf16*)src, n_rows, K, gamma,
                                                            beta, bias_in, bias_out, row_mode);
  else
    launch_k(fold_rows_kernel<float>, cdiv(n_rows, 8), 256, 0, st, (float*)dst, ld_dst, (const float*)src, n_rows, K,
                                                             gamma, beta, bias_in, bias_out, row_mode);
}

void launch_to_f32(cudaStream_t st, int dt, const void* src, float* dst, int n) {
  if (n <= 0) return;
  if (dt == 1) launch_k(to_f32_kernel<bf16>, cdiv(n, 256), 256, 0, st, (const bf16*)src, dst, n);
  else launch_k(to_f32_kernel<float>, cdiv(n, 256), 256, 0, st, (const float*)src, dst, n);
}

void launch_read_kv(cudaStream_t st, int dt, KVCacheView c, int layer0, int seq, int pos0, int n_pos, void* ko,
                    void* vo) {
  if (n_pos <= 0) return;
  if (dt == 1) launch_k(read_kv_kernel<bf16>, n_pos, 256, 0, st, c, layer0, seq, pos0, n_pos, (bf16*)ko, (bf16*)vo);
  else launch_k(read_kv_kernel<float>, n_pos, 256, 0, st, c, layer0, seq, pos0, n_pos, (float*)ko, (float*)vo);
}

// Tile-contiguous weight copy: one thread per 16-byte piece of the destination.  Piece q of
// unit (tile t, k-block kb) sits at chunk c, row r, physical position u; it holds the 8 values of
// row t*32 + r at k = kb*256 + c*64 + (u ^ (r & 7))*8 (the swizzle the stage's 128-byte rows
// carry), zeros past N or K.
__global__ void tile_weight_kernel(const bf16* __restrict__ src, int N, int K, int ld, int nkb, long long pieces,
                                   uint4* __restrict__ dst) {
  const long long q = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= pieces) return;
  const long long unit = q >> 10;           // 1024 pieces of 16 B per unit
  const int w = (int)(q & 1023);
  const int c = w >> 8, r = (w >> 3) & 31, u = w & 7;
  const int t = (int)(unit / nkb), kb = (int)(unit - (long long)t * nkb);
  const int n = t * 32 + r, k = kb * 256 + c * 64 + ((u ^ (r & 7)) << 3);
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (n < N && k < K) v = *reinterpret_cast<const uint4*>(src + (size_t)n * ld + k);   // K % 8 == 0
  dst[q] = v;
}

void launch_tile_weight(cudaStream_t st, const void* src, int N, int K, int ld, void* dst) {
  const int nkb = cdiv(K, TW_KB);
  const long long pieces = (long long)cdiv(N, TW_ROWS) * nkb * (TW_UNIT / 16);
  const int threads = 256;
  tile_weight_kernel<<<(unsigned)((pieces + threads - 1) / threads), threads, 0, st>>>((const bf16*)src, N, K, ld, nkb,
                                                                                       pieces, (uint4*)dst);
}

ADEPT_KTRACE_ATTACH(misc)

}  // namespace adept

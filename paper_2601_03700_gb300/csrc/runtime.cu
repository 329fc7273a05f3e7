// Host runtime of the ADEPT library: model loading and weight repacking, the paged KV
// pool, the early-exit layer loop of prefill / decode, the skipped-layer fill entry
// point, and the C ABI of include/adept.h.
#include "adept.h"
#include "common.cuh"
#include "kernels.h"
#include "gemm_tc.h"
#include "gemm_decode.h"
#include "gemm_stream.h"
#include "model_view.h"
#include "hsm_train.h"

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <random>
#include <string>
#include <unordered_map>
#include <vector>

using namespace adept;

namespace adept {
thread_local bool g_pdl = false;
thread_local SpanCtx g_span = {nullptr, 0};
}

namespace {
thread_local std::string g_load_error;
}

struct LayerW {
  void* w_qkv = nullptr;  // [D_q + 2 D_kv, D]: Q rows, then K rows, then V rows (input-norm gain folded in)
  float* b_qkv = nullptr;
  void* w_o = nullptr;    // [D, D_q]
  float* b_o = nullptr;
  void* w_up = nullptr;   // LLAMA: [2F, D] gate/up interleaved by 16 rows; else [F, D]
  float* b_up = nullptr;
  int up_rows = 0;
  void* w_down = nullptr; // [D, F]
  float* b_down = nullptr;
  float *ln1_g = nullptr, *ln1_b = nullptr, *ln2_g = nullptr, *ln2_b = nullptr;  // post-LN (encoder)
  // tile-contiguous copies for the weight-streaming kernels (bf16 decoders; GemmProblem::Bt)
  void *t_qkv = nullptr, *t_o = nullptr, *t_up = nullptr, *t_down = nullptr;
  // cross-attention sublayer (max_src > 0): W_Qc with the LN_c gain / shift folded in, the
  // source K/V projection [2 D_kv, D] (K rows, then V rows), W_Oc
  void *w_cq = nullptr, *w_ckv = nullptr, *w_co = nullptr;
  float *b_cq = nullptr, *b_ckv = nullptr, *b_co = nullptr;
  void *t_cq = nullptr, *t_co = nullptr;
};

struct ProfRec {
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> ev;
  std::vector<std::pair<double, double>> work;  // (flops, bytes) per recorded launch
};

// HSM training state (adept_hsm_train_*): fp32 master parameters, gradients and AdamW
// moments in flat buffers (parameter i at off[i], each start 64-byte aligned except conv_b,
// which follows conv_w so that the 10 convolution values stay contiguous), transposed weight
// copies for the input-gradient products, and the per-step workspaces.
enum { HT_G0, HT_CONV_W, HT_CONV_B, HT_FC1_W, HT_FC1_B, HT_FC2_W, HT_FC2_B, HT_FC3_W, HT_FC3_B, HT_G1, HT_FC4_W,
       HT_FC4_B, HT_G2, HT_NPARAM };
struct HsmTrain {
  int cap = 0, ldTc = 0, Vp = 0, Vl = 0, part_cols = 0, sms = 1;
  long long step = 0;
  long long off[HT_NPARAM + 1] = {};
  long long numel[HT_NPARAM] = {};
  std::vector<void*> mine;   // this state's allocations (also listed in the model's)
  float *theta = nullptr, *grad = nullptr, *mom1 = nullptr, *mom2 = nullptr;
  void *w1T = nullptr, *w2T = nullptr, *w3T = nullptr, *w4T = nullptr, *headT = nullptr;
  int* iota = nullptr;
  float *c0f = nullptr, *z1f = nullptr, *h1f = nullptr, *z2f = nullptr, *h3f = nullptr, *h5f = nullptr,
        *stf = nullptr, *logits = nullptr, *lossr = nullptr, *dxh = nullptr, *dc0f = nullptr, *dh5f = nullptr,
        *dh4f = nullptr, *dh3f = nullptr, *dh2f = nullptr, *r1 = nullptr, *r2 = nullptr, *cw = nullptr,
        *part = nullptr;
  void *c0t = nullptr, *c0T = nullptr, *h1t = nullptr, *h1T = nullptr, *h2t = nullptr, *h2T = nullptr,
       *h4t = nullptr, *h4T = nullptr, *xht = nullptr, *dlt = nullptr, *dh5t = nullptr, *dh5T = nullptr,
       *dh3t = nullptr, *dh3T = nullptr, *dz2t = nullptr, *dz2T = nullptr;
  // encoders (classification): pooler weight transposed, pooler pre-activations, their
  // gradient, the classifier rows' losses
  void *poolT = nullptr, *dpt = nullptr;
  float *zp = nullptr, *lossc = nullptr;
};

struct adept_model {
  adept_config cfg{};
  int N = 0, D = 0, H = 0, Hkv = 0, dh = 0, Dq = 0, Dkv = 0, F = 0, V = 0, m1 = 0, m2 = 0, dt = 0;
  size_t esz = 4;
  std::vector<void*> allocs;
  std::string err;
  // weights
  void* tok_emb = nullptr;
  void* pos_emb = nullptr;
  float* type_emb = nullptr;
  float *emb_g = nullptr, *emb_b = nullptr;
  std::vector<LayerW> L;
  void* w_head = nullptr;
  float* b_head = nullptr;
  void *w_pool = nullptr, *w_cls = nullptr;
  float *b_pool = nullptr, *b_cls = nullptr;
  float *hsm_g0 = nullptr, *hsm_conv = nullptr, *hsm_g1 = nullptr, *hsm_g2 = nullptr;
  float *hsm_b1 = nullptr, *hsm_b2 = nullptr, *hsm_b3 = nullptr, *hsm_b4 = nullptr;
  void *hsm_w1 = nullptr, *hsm_w2 = nullptr, *hsm_w3 = nullptr, *hsm_w4 = nullptr;
  // tile-contiguous copies of the head and the mapper's FC weights (bf16 decoders)
  void *t_head = nullptr, *t_hsm1 = nullptr, *t_hsm2 = nullptr, *t_hsm3 = nullptr, *t_hsm4 = nullptr;
  float2* rope_table = nullptr;
  // paged KV cache
  void *k_pool = nullptr, *v_pool = nullptr;
  int n_blocks = 0, max_blocks_per_seq = 0;
  int* d_block_table = nullptr;
  std::vector<int> h_block_table, free_list, h_seq_len;
  std::vector<std::vector<int>> seq_blocks;
  int* d_seq_len = nullptr;
  // source cache of the cross-attention (max_src > 0): per layer, max_src positions per
  // sequence in 16-position blocks (sequence b owns blocks b * cs_blocks_per_seq ...)
  void *ck_pool = nullptr, *cv_pool = nullptr;
  int cs_blocks_per_seq = 0;
  int* d_cblock_table = nullptr;
  int* d_src_len = nullptr;          // source positions per sequence (0: not set)
  std::vector<int> h_src_len;
  int *cs_seq = nullptr, *cs_pos = nullptr, *cs_iota = nullptr;   // source row -> (sequence, position)
  void* cs_x = nullptr;              // source states in the GEMM input type
  // pass workspaces (T_max rows)
  int T_max = 0;
  float *X_in[2] = {nullptr, nullptr}, *X_out = nullptr, *I[2] = {nullptr, nullptr};
  int *row_tok[2] = {nullptr, nullptr}, *tok_seq = nullptr, *tok_pos = nullptr, *flag = nullptr, *dst = nullptr;
  float* inv_norm = nullptr;
  float *hsm_s = nullptr, *hsm_prev = nullptr, *hsm_I = nullptr;
  int* exit_tok = nullptr;
  void *xn = nullptr, *q = nullptr, *att = nullptr, *hbuf = nullptr, *xfill = nullptr;
  float *c0f = nullptr, *h1f = nullptr, *h3f = nullptr, *h5f = nullptr;
  void *c0t = nullptr, *h1t = nullptr, *h2t = nullptr, *h4t = nullptr;
  float* final_ = nullptr;
  int* ctr = nullptr;
  unsigned* err_word = nullptr;
  int* head_rows = nullptr;
  void* xhead = nullptr;
  void* pool_t = nullptr;
  float* logits_ws = nullptr;
  float* attn_ws = nullptr;
  int* attn_ctr = nullptr;       // generation-step attention arrival counters (zero between launches)
  int32_t* calib_exit = nullptr; // threshold calibration: exit layers of a calibration pass
  // standardisation statistics of X_out handed from the O projection to the FFN input
  float2* tile_stats = nullptr;                // [DG_MAX_M][D / 32] (mean, M2) of X_out tiles
  // stream-K weight-streaming GEMM workspace (bf16 models): partial tiles and arrival counters
  float* ds_part = nullptr;
  int* ds_cnt = nullptr;
  int ds_ctas = 0;
  float* amax_v = nullptr;       // argmax partials
  int* amax_i = nullptr;
  float* scratch = nullptr;
  size_t scratch_elems = 0;
  // skipped-layer fill workspace (adept_skip_kv_fill)
  int fill_cap = 0;
  void* fill_x = nullptr;
  int *fill_tok = nullptr, *fill_hist = nullptr, *fill_start = nullptr, *fill_cursor = nullptr;
  // generation-step staging buffers (the captured graph reads and writes only these)
  float* d_delta = nullptr;
  int *dec_tok = nullptr, *dec_forced = nullptr, *dec_exit = nullptr, *dec_next = nullptr;
  float* dec_sim = nullptr;
  cudaStream_t cap_stream = nullptr;
  std::vector<cudaGraphExec_t> dec_graph;   // per batch size
  std::vector<int> dec_warm;                // direct runs done per batch size
  // options / instrumentation
  int hsm_identity = 0, profile = 0, force_simt = 0, use_graph = 1, use_dg = 1, use_stream = 1, use_tiled = 1;
  int use_attn_tc = 1;   // prompt-pass attention on the tcgen05 kernel
  int use_fused_exit = 1;   // generation steps: layer i's exit step inside layer i+1's QKV launch
  int exit_metric = 0;   // EXIT_GLOBAL / EXIT_LOCAL / EXIT_BOTH
  int all_at_once = 0;   // prompt passes: sequences leave with their last prompt token
  int stop_entirely = 0; // encoders: exited tokens get no deeper K/V and leave deeper attention
  int32_t* tok_exit = nullptr;   // stop-entirely passes: each token's exit layer so far
  HsmTrain* ht = nullptr;   // HSM training state (adept_hsm_train_init)
  bool xhead_ready = false; // the last generation step left its head input rows in xhead
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  int gemm_cls = ADEPT_PROF_GEMM_PREFILL;
  int last_rows = 0;
  int64_t launches = 0;
  adept_status deferred = ADEPT_OK;   // an error met inside a launch sequence, reported by check_launch
  int64_t graph_launches = 0;   // kernels in one captured generation step
  ProfRec prof[ADEPT_PROF_NCLASS];
  // in-situ spans of the weight-streaming launches (ADEPT_OPT_SPAN_TIMER)
  int span_on = 0;
  SpanSite* span_sites = nullptr;   // SPAN_SITES launch sites, taken in turn (a pass uses fewer)
  SpanTotal* span_tot = nullptr;    // per kernel class
  unsigned span_next = 0;
  unsigned span_in_pass = 0;        // sites taken since the last collect (at most SPAN_SITES)
};
constexpr unsigned SPAN_SITES = 1024;

// ---------------------------------------------------------------------------
// small helpers
// ---------------------------------------------------------------------------
static adept_status fail(adept_model* m, adept_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (m) m->err = buf;
  else g_load_error = buf;
  return s;
}

#define CUDA_TRY(m, call)                                                                               \
  do {                                                                                                  \
    cudaError_t e_ = (call);                                                                            \
    if (e_ != cudaSuccess) return fail(m, ADEPT_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_)); \
  } while (0)

// Allocation-failure hook (adept_set_alloc_fail_after): allocations left before every device
// allocation of the library fails; negative: off.
static std::atomic<long long> g_alloc_budget{-1};

static adept_status dalloc(adept_model* m, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) return ADEPT_OK;
  for (long long b = g_alloc_budget.load(); b >= 0;) {
    if (b == 0) return fail(m, ADEPT_ERR_OOM, "cudaMalloc(%zu) refused by the allocation-failure hook", bytes);
    if (g_alloc_budget.compare_exchange_weak(b, b - 1)) break;
  }
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return fail(m, ADEPT_ERR_OOM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  }
  m->allocs.push_back(*p);
  return ADEPT_OK;
}

template <typename P>
static adept_status dalloc_t(adept_model* m, P** p, size_t count, size_t esz = sizeof(P)) {
  return dalloc(m, (void**)p, count * esz);
}

#define TRY(x)                        \
  do {                                \
    adept_status s_ = (x);            \
    if (s_ != ADEPT_OK) return s_;    \
  } while (0)

static void drop_graphs(adept_model* m) {
  for (auto& g : m->dec_graph)
    if (g) cudaGraphExecDestroy(g);
  for (auto& g : m->dec_graph) g = nullptr;
  for (auto& w : m->dec_warm) w = 0;
}

static void free_all(adept_model* m) {
  drop_graphs(m);
  delete m->ht;
  m->ht = nullptr;
  if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
  m->cap_stream = nullptr;
  for (void* p : m->allocs) cudaFree(p);
  m->allocs.clear();
  for (cudaEvent_t e : m->ev_pool) cudaEventDestroy(e);
  m->ev_pool.clear();
  for (auto& pr : m->prof) pr.ev.clear();
}

static int attn_norm_mode(const adept_model* m) {
  return m->cfg.family == ADEPT_FAMILY_LLAMA ? NORM_RMS : (m->cfg.family == ADEPT_FAMILY_GPT2 ? NORM_LN : NORM_COPY);
}

static KVCacheView cache_view(const adept_model* m) {
  KVCacheView c;
  c.k = m->k_pool;
  c.v = m->v_pool;
  c.block_table = m->d_block_table;
  c.max_blocks_per_seq = m->max_blocks_per_seq;
  c.n_blocks = m->n_blocks;
  c.n_kv_heads = m->Hkv;
  c.head_dim = m->dh;
  c.block_tokens = m->cfg.kv_block_tokens;
  c.max_batch = m->cfg.max_batch;
  return c;
}

static KVCacheView cross_view(const adept_model* m) {
  KVCacheView c;
  c.k = m->ck_pool;
  c.v = m->cv_pool;
  c.block_table = m->d_cblock_table;
  c.max_blocks_per_seq = m->cs_blocks_per_seq;
  c.n_blocks = m->cfg.max_batch * m->cs_blocks_per_seq;
  c.n_kv_heads = m->Hkv;
  c.head_dim = m->dh;
  c.block_tokens = m->cfg.kv_block_tokens;
  c.max_batch = m->cfg.max_batch;
  return c;
}

static Epi epi_base() {
  Epi e;
  memset(&e, 0, sizeof e);
  return e;
}

// ---------------------------------------------------------------------------
// GEMM dispatch: tcgen05 grouped GEMM for bf16 models, SIMT otherwise.
// ---------------------------------------------------------------------------
// Profiling: CUDA events from a pool, recorded on the launching stream around a launch.
static cudaEvent_t pool_event(adept_model* m) {
  if (m->ev_used == m->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    m->ev_pool.push_back(e);
  }
  return m->ev_pool[m->ev_used++];
}
static void prof_begin(adept_model* m, int cls, cudaStream_t st, cudaEvent_t* b) {
  *b = nullptr;
  if (!m->profile) return;
  *b = pool_event(m);
  if (*b) cudaEventRecord(*b, st);
  (void)cls;
}
static void prof_end(adept_model* m, int cls, cudaStream_t st, cudaEvent_t b, double flops, double bytes) {
  if (!m->profile || !b) return;
  cudaEvent_t e = pool_event(m);
  if (!e) return;
  cudaEventRecord(e, st);
  m->prof[cls].ev.push_back({b, e});
  m->prof[cls].work.push_back({flops, bytes});
}

// The SIMT path stages C in fp32 scratch: make room for `elems` floats.
static bool ensure_scratch(adept_model* m, size_t elems) {
  if (elems <= m->scratch_elems) return true;
  if (m->scratch) {
    cudaFree(m->scratch);
    m->allocs.erase(std::remove(m->allocs.begin(), m->allocs.end(), (void*)m->scratch), m->allocs.end());
    m->scratch = nullptr;
    m->scratch_elems = 0;
  }
  if (dalloc_t(m, &m->scratch, elems) != ADEPT_OK) return false;
  m->scratch_elems = elems;
  return true;
}

// Grouped skipped-layer fills take the weight-streaming kernel up to one 8-row block of tokens
// (measured at Llama-7B layer shapes: 1 token at 0.90 of the fill roofline against 0.54 on the
// tcgen05 path, but 16 tokens at 0.36 against 0.54, each CTA then staging a 64 KB operand slice).
constexpr int DG_FILL_MAX_ROWS = 8;

// The generation-step GEMM (gemm_decode.cu) takes single problems of at most DG_MAX_M rows.
static bool dg_takes(const adept_model* m, int n_probs, const GemmProblem& p, int max_rows, const DgNorm* norm) {
  return m->dt == ADEPT_DTYPE_BF16 && !m->force_simt && m->use_dg && n_probs == 1 &&
         decode_gemm_supported(p, max_rows, norm);
}

static DsWork ds_work(const adept_model* m) {
  DsWork w;
  w.part = m->use_stream ? m->ds_part : nullptr;
  w.part_ctas = m->ds_ctas;
  w.cnt = m->ds_cnt;
  w.cnt_cap = DS_CNT_CAP;
  return w;
}

// Sets g_span for the weight-streaming launch of one call (class cls) while the span timer
// is on; consecutive launches take different sites.
struct SpanGuard {
  SpanCtx prev;
  SpanGuard(adept_model* m, int cls) : prev(g_span) {
    if (m->span_on && m->span_sites && m->span_in_pass < SPAN_SITES) {
      // a site is used once between two collects (a pass with more launches records its first
      // SPAN_SITES only)
      g_span = SpanCtx{m->span_sites + (m->span_next++ % SPAN_SITES), cls};
      m->span_in_pass += 1;
    } else {
      g_span = SpanCtx{nullptr, 0};
    }
  }
  ~SpanGuard() { g_span = prev; }
  SpanGuard(const SpanGuard&) = delete;
  SpanGuard& operator=(const SpanGuard&) = delete;
};

// A weight-streaming problem of at most DG_MAX_M rows: the stream-K kernel where it takes the
// shape (weights large enough to stream, A rows fitting in shared memory), else the cluster
// K-split kernel.  Returns the launches, or -1 when neither takes it.
// End of a pass with the span timer on: the pass's sites into the class totals.
static void span_collect(adept_model* m, cudaStream_t st) {
  if (!m->span_on || !m->span_sites) return;
  launch_span_collect(st, m->span_sites, (int)SPAN_SITES, m->span_tot, ADEPT_PROF_NCLASS);
  m->launches += 1;
  m->span_in_pass = 0;
}

static int streaming_gemm(adept_model* m, cudaStream_t st, const GemmProblem& p0, int max_rows, const DgNorm* norm,
                          int cls) {
  SpanGuard sg(m, cls);
  GemmProblem p = p0;
  if (!m->use_tiled) p.Bt = nullptr;
  if (stream_gemm(st, p, max_rows, norm, ds_work(m), m->err_word) >= 0) return 1;
  return decode_gemm(st, p, max_rows, norm, m->err_word);
}

// The grouped skipped-layer fill of a few tokens on the weight-streaming kernels.
static int streaming_gemm_grouped(adept_model* m, cudaStream_t st, const GemmProblem* probs0, int n, int max_rows) {
  SpanGuard sg(m, ADEPT_PROF_KV_FILL);
  std::vector<GemmProblem> copy;
  const GemmProblem* probs = probs0;
  if (!m->use_tiled) {
    copy.assign(probs0, probs0 + n);
    for (auto& q : copy) q.Bt = nullptr;
    probs = copy.data();
  }
  if (stream_gemm_grouped(st, probs, n, max_rows, ds_work(m), m->err_word) >= 0) return 1;
  return max_rows <= DG_FILL_MAX_ROWS ? decode_gemm_grouped(st, probs, n, max_rows, m->err_word) : -1;
}

// The QKV product of a generation step with the previous layer's exit step in the same launch
// (stream-K kernel); -1 when that launch does not take it.
static int streaming_gemm_exit(adept_model* m, cudaStream_t st, const GemmProblem& p0, int max_rows,
                               const DsExit& ex, int cls) {
  if (!m->use_stream || !m->use_dg || m->force_simt || m->dt != ADEPT_DTYPE_BF16) return -1;
  cudaEvent_t b = nullptr;
  prof_begin(m, cls, st, &b);
  int r;
  {
    SpanGuard sg(m, cls);
    GemmProblem p = p0;
    if (!m->use_tiled) p.Bt = nullptr;
    r = stream_gemm_exit(st, p, max_rows, ex, ds_work(m), m->err_word);
  }
  prof_end(m, cls, st, b, 0, 0);
  return r;
}

static void gemm(adept_model* m, cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows,
                 int cls, double flops = 0, double bytes = 0) {
  cudaEvent_t b = nullptr;
  prof_begin(m, cls, st, &b);
  if (dg_takes(m, n_probs, probs[0], max_rows[0], nullptr) && streaming_gemm(m, st, probs[0], max_rows[0], nullptr, cls) >= 0) {
    m->launches += 1;
    prof_end(m, cls, st, b, flops, bytes);
    return;
  }
  if (m->dt == ADEPT_DTYPE_BF16 && !m->force_simt && tc_gemm_supported()) {
    const int nl = tc_gemm_grouped(st, probs, n_probs, max_rows, m->err_word);
    if (nl >= 0) {
      m->launches += nl;
      prof_end(m, cls, st, b, flops, bytes);
      return;
    }
    // shapes the tensor-core path does not take run on the SIMT path
  }
  {
    for (int i = 0; i < n_probs; ++i) {
      if (!ensure_scratch(m, (size_t)max_rows[i] * probs[i].N)) {
        cudaStreamSynchronize(st);
        if (!ensure_scratch(m, (size_t)max_rows[i] * probs[i].N)) {   // the call returns OOM
          m->deferred = ADEPT_ERR_OOM;
          continue;
        }
      }
      launch_gemm_simt(st, m->dt, probs[i], max_rows[i], m->scratch);
      m->launches += 2;
    }
  }
  prof_end(m, cls, st, b, flops, bytes);
}

// GEMM whose A operand is the standardised rows of X (rows in_rows[r], or r; row length
// p.K).  The generation-step GEMM standardises while it stages the operand (with the row
// statistics its producer computed, when given); otherwise the standardisation runs as its
// own launch into p.A first.
static void gemm_std(adept_model* m, cudaStream_t st, const GemmProblem& p, int max_rows, const float* X, int ldx,
                     const int* in_rows, int mode, float eps, int cls, const float2* row_stats = nullptr,
                     const float2* tile_stats = nullptr) {
  const DgNorm nrm{X, ldx, in_rows, mode, eps, row_stats, tile_stats};
  if (dg_takes(m, 1, p, max_rows, &nrm)) {
    cudaEvent_t b = nullptr;
    prof_begin(m, cls, st, &b);
    if (streaming_gemm(m, st, p, max_rows, &nrm, cls) >= 0) {
      m->launches += 1;
      prof_end(m, cls, st, b, 0, 0);
      return;
    }
    prof_end(m, cls, st, b, 0, 0);   // not launched: an empty interval
  }
  launch_standardize(st, m->dt, X, ldx, in_rows, p.rows, max_rows, p.K, mode, eps, const_cast<void*>(p.A), p.lda);
  m->launches += 1;
  gemm(m, st, &p, 1, &max_rows, cls);
}

// ---------------------------------------------------------------------------
// loading
// ---------------------------------------------------------------------------
struct Loader {
  adept_model* m;
  std::unordered_map<std::string, adept_tensor> t;
  void* staging = nullptr;
  size_t staging_bytes = 0;
  float* fstage[2] = {nullptr, nullptr};
  size_t fstage_n = 0;
  cudaStream_t st;

  adept_status find(const std::string& name, int64_t numel, const void** out) {
    auto it = t.find(name);
    if (it == t.end()) return fail(m, ADEPT_ERR_INVALID_ARG, "weight '%s' missing", name.c_str());
    if (it->second.numel != numel)
      return fail(m, ADEPT_ERR_INVALID_ARG, "weight '%s' has %lld elements, expected %lld", name.c_str(),
                  (long long)it->second.numel, (long long)numel);
    if (!it->second.data) return fail(m, ADEPT_ERR_INVALID_ARG, "weight '%s' has a NULL pointer", name.c_str());
    *out = it->second.data;
    return ADEPT_OK;
  }
  bool has(const std::string& name) const { return t.count(name) != 0; }

  // Model-dtype tensor copied verbatim into new device memory.
  adept_status upload(const std::string& name, int64_t numel, void** out) {
    const void* src;
    TRY(find(name, numel, &src));
    TRY(dalloc(m, out, numel * m->esz));
    CUDA_TRY(m, cudaMemcpyAsync(*out, src, numel * m->esz, cudaMemcpyDefault, st));
    return ADEPT_OK;
  }
  // Model-dtype tensor into the staging buffer (device).
  adept_status stage(const std::string& name, int64_t numel, const void** out) {
    const void* src;
    TRY(find(name, numel, &src));
    CUDA_TRY(m, cudaMemcpyAsync(staging, src, numel * m->esz, cudaMemcpyDefault, st));
    *out = staging;
    return ADEPT_OK;
  }
  // Vector converted to fp32 in new device memory (or into `dst` if given).
  adept_status vec_f32(const std::string& name, int64_t n, float** out) {
    const void* src;
    TRY(stage(name, n, &src));
    TRY(dalloc_t(m, out, n));
    launch_to_f32(st, m->dt, src, *out, (int)n);
    CUDA_TRY(m, cudaStreamSynchronize(st));
    return ADEPT_OK;
  }
  adept_status vec_f32_opt(const std::string& name, int64_t n, float** out) {
    if (!has(name)) {
      TRY(dalloc_t(m, out, n));
      CUDA_TRY(m, cudaMemsetAsync(*out, 0, n * sizeof(float), st));
      return ADEPT_OK;
    }
    return vec_f32(name, n, out);
  }
  // fp32 copy of a vector into a reusable slot (gains / shifts used only while folding).
  adept_status tmp_f32(const std::string& name, int64_t n, int slot, float** out) {
    const void* src;
    TRY(stage(name, n, &src));
    launch_to_f32(st, m->dt, src, fstage[slot], (int)n);
    CUDA_TRY(m, cudaStreamSynchronize(st));
    *out = fstage[slot];
    return ADEPT_OK;
  }
  // rows of `name` ([n_rows, K]) folded with gain/shift into dst (ld K) at row offset.
  adept_status fold(const std::string& name, int n_rows, int K, void* dst, int row_off, const float* gamma,
                    const float* beta, const float* bias_in, float* bias_out, int row_mode = 0) {
    const void* src;
    TRY(stage(name, (int64_t)n_rows * K, &src));
    launch_fold_rows(st, m->dt, (char*)dst + (size_t)row_off * K * m->esz, K, src, n_rows, K, gamma, beta, bias_in,
                     bias_out ? bias_out + row_off : nullptr, row_mode);
    CUDA_TRY(m, cudaStreamSynchronize(st));
    return ADEPT_OK;
  }
};

static adept_status validate_cfg(adept_config* c) {
  if (c->n_kv_heads == 0) c->n_kv_heads = c->n_heads;
  if (c->family < 0 || c->family > 2) return fail(nullptr, ADEPT_ERR_INVALID_ARG, "family %d unknown", c->family);
  if (c->dtype != ADEPT_DTYPE_F32 && c->dtype != ADEPT_DTYPE_BF16)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "dtype %d unknown", c->dtype);
  if (c->n_layers < 1 || c->d_model < 1 || c->n_heads < 1 || c->d_ffn < 1 || c->vocab < 1)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "non-positive model size");
  if (c->head_dim != 32 && c->head_dim != 64 && c->head_dim != 128)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "head_dim %d unsupported (32, 64 or 128)", c->head_dim);
  if (c->n_heads % c->n_kv_heads) return fail(nullptr, ADEPT_ERR_INVALID_ARG, "n_heads %% n_kv_heads != 0");
  if (c->d_model % 8 || c->d_ffn % 16 || c->hsm_m1 % 8 || c->hsm_m2 % 8)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "d_model, hsm widths must be multiples of 8 and d_ffn of 16");
  if (c->hsm_m1 < 1 || c->hsm_m2 < 1) return fail(nullptr, ADEPT_ERR_INVALID_ARG, "HSM widths must be positive");
  if (c->max_batch < 1 || c->max_seq < 1 || c->kv_block_tokens < 1)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "max_batch, max_seq, kv_block_tokens must be positive");
  if (c->family != ADEPT_FAMILY_LLAMA && c->max_pos < c->max_seq)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "max_pos must cover max_seq for learned positions");
  if (c->family == ADEPT_FAMILY_BERT && c->n_classes < 1)
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "encoder needs n_classes >= 1");
  if ((long long)c->max_batch * c->max_seq > (1LL << 26))
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "max_batch * max_seq too large");
  if (c->max_src < 0 || (c->max_src > 0 && c->family != ADEPT_FAMILY_GPT2))
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "cross-attention (max_src > 0) is defined for GPT-2-family decoders");
  if ((long long)c->max_batch * c->max_src > (1LL << 24))
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "max_batch * max_src too large");
  return ADEPT_OK;
}

static adept_status load_weights(adept_model* m, Loader& ld) {
  const adept_config& c = m->cfg;
  const int D = m->D, F = m->F, V = m->V, Dq = m->Dq, Dkv = m->Dkv, m1 = m->m1, m2 = m->m2;
  const int fam = c.family;
  // staging sized for the largest single tensor
  size_t big = (size_t)V * D;
  big = std::max(big, (size_t)F * D);
  big = std::max(big, (size_t)m1 * m2);
  big = std::max(big, (size_t)std::max(m1, D) * std::max(m1, D));
  big = std::max(big, (size_t)Dq * D);
  if (fam != ADEPT_FAMILY_LLAMA) big = std::max(big, (size_t)c.max_pos * D);
  TRY(dalloc(m, &ld.staging, big * m->esz));
  ld.fstage_n = std::max<size_t>(std::max(D, m1), 16);
  TRY(dalloc_t(m, &ld.fstage[0], ld.fstage_n));
  TRY(dalloc_t(m, &ld.fstage[1], ld.fstage_n));

  TRY(ld.upload("tok_emb", (int64_t)V * D, &m->tok_emb));
  if (fam != ADEPT_FAMILY_LLAMA) TRY(ld.upload("pos_emb", (int64_t)c.max_pos * D, &m->pos_emb));
  if (fam == ADEPT_FAMILY_BERT) {
    TRY(ld.vec_f32("type_emb", D, &m->type_emb));
    TRY(ld.vec_f32("emb_ln.g", D, &m->emb_g));
    TRY(ld.vec_f32("emb_ln.b", D, &m->emb_b));
  }
  m->L.resize(m->N);
  const int nqkv = Dq + 2 * Dkv;
  for (int l = 0; l < m->N; ++l) {
    LayerW& w = m->L[l];
    const std::string p = "layers." + std::to_string(l) + ".";
    TRY(dalloc(m, &w.w_qkv, (size_t)nqkv * D * m->esz));
    TRY(dalloc_t(m, &w.b_qkv, nqkv));
    float *g = nullptr, *b = nullptr, *bin = nullptr;
    if (fam == ADEPT_FAMILY_LLAMA) {
      TRY(ld.tmp_f32(p + "attn_norm.g", D, 0, &g));
    } else if (fam == ADEPT_FAMILY_GPT2) {
      TRY(ld.tmp_f32(p + "attn_norm.g", D, 0, &g));
      TRY(ld.tmp_f32(p + "attn_norm.b", D, 1, &b));
    }
    const char* qn[3] = {"wq", "wk", "wv"};
    const char* bn[3] = {"bq", "bk", "bv"};
    const int rows[3] = {Dq, Dkv, Dkv};
    int off = 0;
    for (int k = 0; k < 3; ++k) {
      bin = nullptr;
      float* btmp = nullptr;
      if (fam != ADEPT_FAMILY_LLAMA) {
        TRY(dalloc_t(m, &btmp, rows[k]));
        const void* src;
        TRY(ld.find(p + bn[k], rows[k], &src));
        // biases go through the second fp32 slot only after the shift was consumed; use a private buffer
        CUDA_TRY(m, cudaMemcpyAsync(ld.staging, src, rows[k] * m->esz, cudaMemcpyDefault, ld.st));
        launch_to_f32(ld.st, m->dt, ld.staging, btmp, rows[k]);
        CUDA_TRY(m, cudaStreamSynchronize(ld.st));
        bin = btmp;
      }
      const int rmode = (fam == ADEPT_FAMILY_LLAMA && k < 2) ? m->dh : 0;  // RoPE pairs made adjacent
      TRY(ld.fold(p + qn[k], rows[k], D, w.w_qkv, off, g, b, bin, w.b_qkv, rmode));
      off += rows[k];
    }
    TRY(ld.upload(p + "wo", (int64_t)D * Dq, &w.w_o));
    TRY(ld.vec_f32_opt(p + "bo", D, &w.b_o));
    float *g2 = nullptr, *b2 = nullptr;
    if (fam == ADEPT_FAMILY_LLAMA) {
      TRY(ld.tmp_f32(p + "ffn_norm.g", D, 0, &g2));
      w.up_rows = 2 * F;
      TRY(dalloc(m, &w.w_up, (size_t)2 * F * D * m->esz));
      TRY(dalloc_t(m, &w.b_up, 2 * F));
      TRY(ld.fold(p + "w_gate", F, D, w.w_up, 0, g2, nullptr, nullptr, w.b_up, 1));
      TRY(ld.fold(p + "w_up", F, D, w.w_up, 0, g2, nullptr, nullptr, w.b_up, 2));
      TRY(ld.upload(p + "w_down", (int64_t)D * F, &w.w_down));
      TRY(ld.vec_f32_opt(p + "b_down_absent", D, &w.b_down));
    } else {
      w.up_rows = F;
      TRY(dalloc(m, &w.w_up, (size_t)F * D * m->esz));
      TRY(dalloc_t(m, &w.b_up, F));
      float* bfc = nullptr;
      TRY(ld.vec_f32(p + "b_fc", F, &bfc));
      if (fam == ADEPT_FAMILY_GPT2) {
        TRY(ld.tmp_f32(p + "ffn_norm.g", D, 0, &g2));
        TRY(ld.tmp_f32(p + "ffn_norm.b", D, 1, &b2));
      }
      TRY(ld.fold(p + "w_fc", F, D, w.w_up, 0, g2, b2, bfc, w.b_up));
      TRY(ld.upload(p + "w_proj", (int64_t)D * F, &w.w_down));
      TRY(ld.vec_f32(p + "b_proj", D, &w.b_down));
      if (fam == ADEPT_FAMILY_BERT) {
        TRY(ld.vec_f32(p + "attn_norm.g", D, &w.ln1_g));
        TRY(ld.vec_f32(p + "attn_norm.b", D, &w.ln1_b));
        TRY(ld.vec_f32(p + "ffn_norm.g", D, &w.ln2_g));
        TRY(ld.vec_f32(p + "ffn_norm.b", D, &w.ln2_b));
      }
    }
    if (c.max_src > 0) {
      // cross-attention: LN_c folded into W_Qc (like the layer's input norm into W_qkv)
      float *cbq = nullptr, *cbk = nullptr, *cbv = nullptr, *cg = nullptr, *cb = nullptr;
      TRY(ld.vec_f32(p + "cbq", Dq, &cbq));
      TRY(ld.vec_f32(p + "cbk", Dkv, &cbk));
      TRY(ld.vec_f32(p + "cbv", Dkv, &cbv));
      TRY(ld.tmp_f32(p + "cross_norm.g", D, 0, &cg));
      TRY(ld.tmp_f32(p + "cross_norm.b", D, 1, &cb));
      TRY(dalloc(m, &w.w_cq, (size_t)Dq * D * m->esz));
      TRY(dalloc_t(m, &w.b_cq, Dq));
      TRY(ld.fold(p + "cwq", Dq, D, w.w_cq, 0, cg, cb, cbq, w.b_cq));
      TRY(dalloc(m, &w.w_ckv, (size_t)2 * Dkv * D * m->esz));
      TRY(dalloc_t(m, &w.b_ckv, 2 * Dkv));
      TRY(ld.fold(p + "cwk", Dkv, D, w.w_ckv, 0, nullptr, nullptr, cbk, w.b_ckv));
      TRY(ld.fold(p + "cwv", Dkv, D, w.w_ckv, Dkv, nullptr, nullptr, cbv, w.b_ckv));
      TRY(ld.upload(p + "cwo", (int64_t)D * Dq, &w.w_co));
      TRY(ld.vec_f32(p + "cbo", D, &w.b_co));
    }
  }
  // output heads (final norm gain / shift folded into the head)
  if (fam == ADEPT_FAMILY_LLAMA) {
    float* g = nullptr;
    TRY(ld.tmp_f32("final_norm.g", D, 0, &g));
    TRY(dalloc(m, &m->w_head, (size_t)V * D * m->esz));
    TRY(dalloc_t(m, &m->b_head, V));
    TRY(ld.fold("lm_head", V, D, m->w_head, 0, g, nullptr, nullptr, m->b_head));
  } else if (fam == ADEPT_FAMILY_GPT2) {
    float *g = nullptr, *b = nullptr;
    TRY(ld.tmp_f32("final_norm.g", D, 0, &g));
    TRY(ld.tmp_f32("final_norm.b", D, 1, &b));
    TRY(dalloc(m, &m->w_head, (size_t)V * D * m->esz));
    TRY(dalloc_t(m, &m->b_head, V));
    TRY(ld.fold("tok_emb", V, D, m->w_head, 0, g, b, nullptr, m->b_head));
  } else {
    TRY(ld.upload("pool.w", (int64_t)D * D, &m->w_pool));
    TRY(ld.vec_f32("pool.b", D, &m->b_pool));
    TRY(ld.upload("cls.w", (int64_t)c.n_classes * D, &m->w_cls));
    TRY(ld.vec_f32("cls.b", c.n_classes, &m->b_cls));
  }
  // Hidden State Mapper (App. B Table S1)
  TRY(ld.vec_f32("hsm.g0", D, &m->hsm_g0));
  TRY(dalloc_t(m, &m->hsm_conv, 10));
  {
    const void* src;
    TRY(ld.stage("hsm.conv_w", 9, &src));
    launch_to_f32(ld.st, m->dt, src, m->hsm_conv, 9);
    CUDA_TRY(m, cudaStreamSynchronize(ld.st));
    TRY(ld.stage("hsm.conv_b", 1, &src));
    launch_to_f32(ld.st, m->dt, src, m->hsm_conv + 9, 1);
    CUDA_TRY(m, cudaStreamSynchronize(ld.st));
  }
  TRY(ld.upload("hsm.fc1_w", (int64_t)m1 * D, &m->hsm_w1));
  TRY(ld.vec_f32("hsm.fc1_b", m1, &m->hsm_b1));
  TRY(ld.upload("hsm.fc2_w", (int64_t)m2 * m1, &m->hsm_w2));
  TRY(ld.vec_f32("hsm.fc2_b", m2, &m->hsm_b2));
  TRY(ld.upload("hsm.fc3_w", (int64_t)m1 * m2, &m->hsm_w3));
  TRY(ld.vec_f32("hsm.fc3_b", m1, &m->hsm_b3));
  TRY(ld.vec_f32("hsm.g1", m1, &m->hsm_g1));
  TRY(ld.upload("hsm.fc4_w", (int64_t)D * m1, &m->hsm_w4));
  TRY(ld.vec_f32("hsm.fc4_b", D, &m->hsm_b4));
  TRY(ld.vec_f32("hsm.g2", D, &m->hsm_g2));
  CUDA_TRY(m, cudaStreamSynchronize(ld.st));
  return ADEPT_OK;
}

static adept_status alloc_runtime(adept_model* m) {
  const adept_config& c = m->cfg;
  const int D = m->D, T = m->T_max;
  // RoPE table (cos, sin) per position and pair, evaluated in double once.
  if (c.family == ADEPT_FAMILY_LLAMA) {
    const int half = m->dh / 2;
    // every position a reserved KV block can hold (max_seq rounded up to whole blocks)
    const int rope_rows = cdiv(c.max_seq, c.kv_block_tokens) * c.kv_block_tokens;
    std::vector<float2> tab((size_t)rope_rows * half);
    for (int p = 0; p < rope_rows; ++p)
      for (int i = 0; i < half; ++i) {
        const double inv = std::pow((double)c.rope_theta, -2.0 * i / m->dh);
        const double a = p * inv;
        tab[(size_t)p * half + i] = make_float2((float)std::cos(a), (float)std::sin(a));
      }
    TRY(dalloc_t(m, &m->rope_table, tab.size()));
    CUDA_TRY(m, cudaMemcpy(m->rope_table, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice));
  }
  // paged KV pool
  m->max_blocks_per_seq = cdiv(c.max_seq, c.kv_block_tokens);
  m->n_blocks = c.kv_pool_blocks > 0 ? c.kv_pool_blocks : c.max_batch * m->max_blocks_per_seq;
  const size_t per_layer = (size_t)m->n_blocks * m->Hkv * c.kv_block_tokens * m->dh;
  TRY(dalloc(m, &m->k_pool, per_layer * m->N * m->esz));
  TRY(dalloc(m, &m->v_pool, per_layer * m->N * m->esz));
  m->h_block_table.assign((size_t)c.max_batch * m->max_blocks_per_seq, -1);
  TRY(dalloc_t(m, &m->d_block_table, m->h_block_table.size()));
  CUDA_TRY(m, cudaMemcpy(m->d_block_table, m->h_block_table.data(), m->h_block_table.size() * sizeof(int),
                         cudaMemcpyHostToDevice));
  m->free_list.resize(m->n_blocks);
  for (int i = 0; i < m->n_blocks; ++i) m->free_list[i] = m->n_blocks - 1 - i;  // pop_back hands out 0, 1, ...
  if (c.block_shuffle_seed) {
    std::mt19937_64 rng(c.block_shuffle_seed);
    std::shuffle(m->free_list.begin(), m->free_list.end(), rng);
  }
  m->seq_blocks.assign(c.max_batch, {});
  m->h_seq_len.assign(c.max_batch, 0);
  TRY(dalloc_t(m, &m->d_seq_len, c.max_batch));
  CUDA_TRY(m, cudaMemset(m->d_seq_len, 0, c.max_batch * sizeof(int)));
  if (c.max_src > 0) {
    // source cache: every sequence owns its blocks (b * per_seq + k), so the table is fixed
    m->cs_blocks_per_seq = cdiv(c.max_src, c.kv_block_tokens);
    const int nb = c.max_batch * m->cs_blocks_per_seq;
    const size_t cper = (size_t)nb * m->Hkv * c.kv_block_tokens * m->dh;
    TRY(dalloc(m, &m->ck_pool, cper * m->N * m->esz));
    TRY(dalloc(m, &m->cv_pool, cper * m->N * m->esz));
    std::vector<int> tab(nb), iota((size_t)c.max_batch * c.max_src);
    for (int i = 0; i < nb; ++i) tab[i] = i;
    for (size_t i = 0; i < iota.size(); ++i) iota[i] = (int)i;
    TRY(dalloc_t(m, &m->d_cblock_table, nb));
    CUDA_TRY(m, cudaMemcpy(m->d_cblock_table, tab.data(), nb * sizeof(int), cudaMemcpyHostToDevice));
    TRY(dalloc_t(m, &m->cs_iota, iota.size()));
    CUDA_TRY(m, cudaMemcpy(m->cs_iota, iota.data(), iota.size() * sizeof(int), cudaMemcpyHostToDevice));
    TRY(dalloc_t(m, &m->cs_seq, iota.size()));
    TRY(dalloc_t(m, &m->cs_pos, iota.size()));
    TRY(dalloc(m, &m->cs_x, iota.size() * D * m->esz));
    TRY(dalloc_t(m, &m->d_src_len, c.max_batch));
    CUDA_TRY(m, cudaMemset(m->d_src_len, 0, c.max_batch * sizeof(int)));
    m->h_src_len.assign(c.max_batch, 0);
  }
  // pass workspaces
  const size_t TD = (size_t)T * D;
  for (int k = 0; k < 2; ++k) {
    TRY(dalloc_t(m, &m->X_in[k], TD));
    TRY(dalloc_t(m, &m->I[k], TD));
    TRY(dalloc_t(m, &m->row_tok[k], T));
  }
  TRY(dalloc_t(m, &m->X_out, TD));
  TRY(dalloc_t(m, &m->tok_seq, T));
  TRY(dalloc_t(m, &m->tok_pos, T));
  TRY(dalloc_t(m, &m->flag, T));
  TRY(dalloc_t(m, &m->dst, T));
  TRY(dalloc_t(m, &m->inv_norm, T));
  TRY(dalloc_t(m, &m->hsm_s, TD));
  TRY(dalloc_t(m, &m->hsm_prev, TD));
  TRY(dalloc_t(m, &m->hsm_I, TD));
  TRY(dalloc_t(m, &m->exit_tok, T));
  TRY(dalloc_t(m, &m->final_, TD));
  TRY(dalloc(m, &m->xn, TD * m->esz));
  TRY(dalloc(m, &m->q, (size_t)T * m->Dq * m->esz));
  TRY(dalloc(m, &m->att, (size_t)T * m->Dq * m->esz));
  TRY(dalloc(m, &m->hbuf, (size_t)T * m->F * m->esz));
  TRY(dalloc(m, &m->xfill, TD * m->esz));
  TRY(dalloc_t(m, &m->c0f, TD));
  TRY(dalloc(m, &m->c0t, TD * m->esz));
  TRY(dalloc_t(m, &m->h1f, (size_t)T * m->m1));
  TRY(dalloc(m, &m->h1t, (size_t)T * m->m1 * m->esz));
  TRY(dalloc(m, &m->h2t, (size_t)T * m->m2 * m->esz));
  TRY(dalloc_t(m, &m->h3f, (size_t)T * m->m1));
  TRY(dalloc(m, &m->h4t, (size_t)T * m->m1 * m->esz));
  TRY(dalloc_t(m, &m->h5f, TD));
  TRY(dalloc_t(m, &m->ctr, ctr_words(m->N)));
  TRY(dalloc_t(m, &m->err_word, 1));
  CUDA_TRY(m, cudaMemset(m->err_word, 0, sizeof(unsigned)));
  TRY(dalloc_t(m, &m->head_rows, c.max_batch));
  TRY(dalloc(m, &m->xhead, (size_t)c.max_batch * D * m->esz));
  TRY(dalloc(m, &m->pool_t, (size_t)c.max_batch * D * m->esz));
  const int nout = c.family == ADEPT_FAMILY_BERT ? c.n_classes : m->V;
  TRY(dalloc_t(m, &m->logits_ws, (size_t)c.max_batch * nout));
  TRY(dalloc_t(m, &m->attn_ws, (size_t)c.max_batch * m->H * ATTN_MAX_SPLIT * (m->dh + 2)));
  TRY(dalloc_t(m, &m->attn_ctr, (size_t)c.max_batch * m->H));
  TRY(dalloc_t(m, &m->tile_stats, (size_t)DG_MAX_M * (m->D / 32 + 1)));
  if (m->dt == ADEPT_DTYPE_BF16) {
    int dev = 0, sms = 0;
    CUDA_TRY(m, cudaGetDevice(&dev));
    CUDA_TRY(m, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    m->ds_ctas = std::max(sms, 1);
    TRY(dalloc(m, (void**)&m->ds_part, stream_gemm_part_bytes(m->ds_ctas)));
    TRY(dalloc_t(m, &m->ds_cnt, DS_CNT_CAP));
    CUDA_TRY(m, cudaMemset(m->ds_cnt, 0, sizeof(int) * DS_CNT_CAP));
  }
  CUDA_TRY(m, cudaMemset(m->attn_ctr, 0, sizeof(int) * c.max_batch * m->H));
  TRY(dalloc_t(m, &m->d_delta, 1));
  TRY(dalloc_t(m, &m->amax_v, (size_t)c.max_batch * 32));
  TRY(dalloc_t(m, &m->amax_i, (size_t)c.max_batch * 32));
  TRY(dalloc_t(m, &m->dec_tok, c.max_batch));
  TRY(dalloc_t(m, &m->dec_forced, c.max_batch));
  TRY(dalloc_t(m, &m->dec_exit, c.max_batch));
  TRY(dalloc_t(m, &m->dec_next, c.max_batch));
  TRY(dalloc_t(m, &m->dec_sim, (size_t)c.max_batch * m->N));
  m->dec_graph.assign(c.max_batch + 1, nullptr);
  m->dec_warm.assign(c.max_batch + 1, 0);
  // SIMT scratch: the widest GEMM output of any pass step
  size_t w = std::max({(size_t)m->Dq + 2 * m->Dkv, (size_t)m->L[0].up_rows, (size_t)m->m1, (size_t)m->m2, (size_t)D});
  m->scratch_elems = std::max(w * T, (size_t)c.max_batch * nout);
  TRY(dalloc_t(m, &m->scratch, m->scratch_elems));
  return ADEPT_OK;
}

// Tile-contiguous copies of the streamed weights (bf16 decoders): every layer projection, the
// LM head and the mapper's four FC matrices, for the weight-streaming kernels of generation
// steps and small fills (contiguous 16 KB units instead of 32 row segments per copy).  The
// row-major weights stay for the tensor-core prompt pass and the mapper's training.
static adept_status tile_into(adept_model* m, cudaStream_t st, const void* src, int N, int K, void** dst) {
  TRY(dalloc(m, dst, tiled_bytes(N, K)));
  launch_tile_weight(st, src, N, K, K, *dst);
  return ADEPT_OK;
}

static adept_status retile_hsm(adept_model* m, cudaStream_t st, bool alloc);
static adept_status make_tiled(adept_model* m, cudaStream_t st) {
  if (m->dt != ADEPT_DTYPE_BF16 || m->cfg.family == ADEPT_FAMILY_BERT) return ADEPT_OK;
  const int D = m->D, Dq = m->Dq, Dkv = m->Dkv, F = m->F;
  for (int l = 0; l < m->N; ++l) {
    LayerW& w = m->L[l];
    TRY(tile_into(m, st, w.w_qkv, Dq + 2 * Dkv, D, &w.t_qkv));
    TRY(tile_into(m, st, w.w_o, D, Dq, &w.t_o));
    TRY(tile_into(m, st, w.w_up, w.up_rows, D, &w.t_up));
    TRY(tile_into(m, st, w.w_down, D, F, &w.t_down));
    if (w.w_cq) {
      TRY(tile_into(m, st, w.w_cq, Dq, D, &w.t_cq));
      TRY(tile_into(m, st, w.w_co, D, Dq, &w.t_co));
    }
  }
  TRY(tile_into(m, st, m->w_head, m->V, D, &m->t_head));
  return retile_hsm(m, st, true);
}

// The mapper's tiled copies from its row-major weights (at load; after every training step).
static adept_status retile_hsm(adept_model* m, cudaStream_t st, bool alloc) {
  if (!alloc && !m->t_hsm1) return ADEPT_OK;
  const int D = m->D, m1 = m->m1, m2 = m->m2;
  if (alloc) {
    TRY(tile_into(m, st, m->hsm_w1, m1, D, &m->t_hsm1));
    TRY(tile_into(m, st, m->hsm_w2, m2, m1, &m->t_hsm2));
    TRY(tile_into(m, st, m->hsm_w3, m1, m2, &m->t_hsm3));
    TRY(tile_into(m, st, m->hsm_w4, D, m1, &m->t_hsm4));
  } else {
    launch_tile_weight(st, m->hsm_w1, m1, D, D, m->t_hsm1);
    launch_tile_weight(st, m->hsm_w2, m2, m1, m1, m->t_hsm2);
    launch_tile_weight(st, m->hsm_w3, m1, m2, m2, m->t_hsm3);
    launch_tile_weight(st, m->hsm_w4, D, m1, m1, m->t_hsm4);
    m->launches += 4;
  }
  return ADEPT_OK;
}

// ---------------------------------------------------------------------------
// sequences and KV blocks
// ---------------------------------------------------------------------------
static adept_status reserve_seqs(adept_model* m, int batch, const int* lens, cudaStream_t st) {
  const adept_config& c = m->cfg;
  for (int b = 0; b < batch; ++b) {
    for (int blk : m->seq_blocks[b]) m->free_list.push_back(blk);
    m->seq_blocks[b].clear();
    for (int k = 0; k < m->max_blocks_per_seq; ++k) m->h_block_table[(size_t)b * m->max_blocks_per_seq + k] = -1;
  }
  for (int b = 0; b < batch; ++b) {
    const int need = m->max_blocks_per_seq;
    if ((int)m->free_list.size() < need)
      return fail(m, ADEPT_ERR_CAPACITY, "KV block pool exhausted (%d free, %d needed)", (int)m->free_list.size(), need);
    for (int k = 0; k < need; ++k) {
      const int blk = m->free_list.back();
      m->free_list.pop_back();
      m->seq_blocks[b].push_back(blk);
      m->h_block_table[(size_t)b * m->max_blocks_per_seq + k] = blk;
    }
    m->h_seq_len[b] = lens[b];
  }
  CUDA_TRY(m, cudaMemcpyAsync(m->d_block_table, m->h_block_table.data(),
                              (size_t)batch * m->max_blocks_per_seq * sizeof(int), cudaMemcpyHostToDevice, st));
  CUDA_TRY(m, cudaMemcpyAsync(m->d_seq_len, m->h_seq_len.data(), batch * sizeof(int), cudaMemcpyHostToDevice, st));
  (void)c;
  return ADEPT_OK;
}

// ---------------------------------------------------------------------------
// the early-exit pass
// ---------------------------------------------------------------------------

// xhead (generation steps): each exit's standardised s~ also becomes its head input row.
static void run_hsm(adept_model* m, cudaStream_t st, DevRange rows, int max_rows, int a_rows, void* xhead = nullptr) {
  const int D = m->D, m1 = m->m1, m2 = m->m2;
  const float eps = m->cfg.hsm_eps;
  if (m->hsm_identity) {
    launch_hsm_out(st, m->dt, nullptr, nullptr, m->hsm_s, 1, rows, max_rows, D, m->hsm_g2, eps, m->exit_tok,
                   m->final_, m->xfill, attn_norm_mode(m), m->cfg.norm_eps, xhead);
    m->launches += 1;
    return;
  }
  launch_hsm_prep(st, m->dt, m->hsm_s, m->hsm_prev, m->hsm_I, rows, max_rows, D, m->hsm_g0, m->hsm_conv, eps, m->c0f,
                  m->c0t);
  m->launches += 1;
  GemmProblem p;
  memset(&p, 0, sizeof p);
  p.rows = rows;
  p.a_rows = a_rows;
  p.split_live = 1;   // the exiting rows of one layer: usually a small part of the pass
  // FC1: h1 = GELU(W1 c0 + b1)
  p.A = m->c0t; p.lda = D; p.B = m->hsm_w1; p.ldb = D; p.N = m1; p.K = D; p.Bt = m->t_hsm1; p.bt_nkb = cdiv(D, TW_KB);
  p.epi = epi_base(); p.epi.kind = EPI_ACT; p.epi.act = ACT_GELU_ERF; p.epi.bias = m->hsm_b1;
  p.epi.out_t = m->h1t; p.epi.ld_t = m1; p.epi.out_f32 = m->h1f; p.epi.ld_f32 = m1;
  gemm(m, st, &p, 1, &max_rows, m->gemm_cls);
  // FC2: h2 = GELU(W2 h1 + b2)
  p.A = m->h1t; p.lda = m1; p.B = m->hsm_w2; p.ldb = m1; p.N = m2; p.K = m1; p.Bt = m->t_hsm2; p.bt_nkb = cdiv(m1, TW_KB);
  p.epi = epi_base(); p.epi.kind = EPI_ACT; p.epi.act = ACT_GELU_ERF; p.epi.bias = m->hsm_b2;
  p.epi.out_t = m->h2t; p.epi.ld_t = m2;
  gemm(m, st, &p, 1, &max_rows, m->gemm_cls);
  // FC3: h3 = W3 h2 + b3
  p.A = m->h2t; p.lda = m2; p.B = m->hsm_w3; p.ldb = m2; p.N = m1; p.K = m2; p.Bt = m->t_hsm3; p.bt_nkb = cdiv(m2, TW_KB);
  p.epi = epi_base(); p.epi.kind = EPI_F32; p.epi.bias = m->hsm_b3; p.epi.out_f32 = m->h3f; p.epi.ld_f32 = m1;
  gemm(m, st, &p, 1, &max_rows, m->gemm_cls);
  launch_hsm_mid(st, m->dt, m->h3f, m->h1f, rows, max_rows, m1, m->hsm_g1, eps, m->h4t);
  m->launches += 1;
  // FC4: h5 = W4 h4 + b4
  p.A = m->h4t; p.lda = m1; p.B = m->hsm_w4; p.ldb = m1; p.N = D; p.K = m1; p.Bt = m->t_hsm4; p.bt_nkb = cdiv(m1, TW_KB);
  p.epi = epi_base(); p.epi.kind = EPI_F32; p.epi.bias = m->hsm_b4; p.epi.out_f32 = m->h5f; p.epi.ld_f32 = D;
  gemm(m, st, &p, 1, &max_rows, m->gemm_cls);
  launch_hsm_out(st, m->dt, m->h5f, m->c0f, m->hsm_s, 0, rows, max_rows, D, m->hsm_g2, eps, m->exit_tok, m->final_,
                 m->xfill, attn_norm_mode(m), m->cfg.norm_eps, xhead);
  m->launches += 1;
}

// KV-only projection problem of layer `layer0` for the rows of `xs` (K-major x~ rows).
static GemmProblem kv_problem(adept_model* m, int layer0, const void* xs, int a_rows, DevRange rows,
                              const int* row_tok, const int* tok_seq, const int* tok_pos) {
  GemmProblem p;
  memset(&p, 0, sizeof p);
  const LayerW& w = m->L[layer0];
  p.A = xs; p.lda = m->D; p.a_rows = a_rows;
  p.B = (const char*)w.w_qkv + (size_t)m->Dq * m->D * m->esz; p.ldb = m->D;
  if (w.t_qkv && m->Dq % TW_ROWS == 0) {   // the K/V rows start at a whole tile of the copy
    p.bt_nkb = cdiv(m->D, TW_KB);
    p.Bt = (const char*)w.t_qkv + (size_t)(m->Dq / TW_ROWS) * p.bt_nkb * TW_UNIT;
  }
  p.rows = rows; p.N = 2 * m->Dkv; p.K = m->D;
  p.epi = epi_base();
  p.epi.kind = EPI_KV; p.epi.bias = w.b_qkv + m->Dq;
  p.epi.row_tok = row_tok; p.epi.tok_seq = tok_seq; p.epi.tok_pos = tok_pos;
  p.epi.cache = cache_view(m); p.epi.layer0 = layer0;
  p.epi.n_q_cols = 0; p.epi.n_kv_cols = m->Dkv; p.epi.head_dim = m->dh;
  p.epi.rope = m->cfg.family == ADEPT_FAMILY_LLAMA; p.epi.rope_table = m->rope_table;
  return p;
}

// One early-exit pass over n_tok tokens.  The threshold delta is read from m->d_delta
// (device memory), so a captured generation step does not depend on it.
static adept_status run_pass(adept_model* m, int n_tok, int batch, int prompt_len, bool decode, const int32_t* tokens,
                             const int32_t* forced, int32_t* exit_out, float* sim_out, cudaStream_t st) {
  m->gemm_cls = decode ? ADEPT_PROF_GEMM_DECODE : ADEPT_PROF_GEMM_PREFILL;
  const adept_config& c = m->cfg;
  const int N = m->N, D = m->D, Dq = m->Dq, Dkv = m->Dkv;
  const int fam = c.family;
  const int amode = attn_norm_mode(m);
  const float eps = c.norm_eps;
  m->last_rows = n_tok;
  // encoder "stop entirely" (Sec. 4.3, downstream tasks): exits are recorded in tok_exit
  // (the attention leaves out keys of tokens gone before its layer) and get no fills
  const bool stop = fam == ADEPT_FAMILY_BERT && m->stop_entirely && !decode;
  const bool cross = c.max_src > 0;   // encoder-decoder decoder: a cross-attention sublayer per layer
  // generation steps of bf16 decoders: the producers of the final states (the last layer's
  // row scatter, the HSM's output step) also write them standardised for the head, so the
  // head GEMM streams its weights against ready bf16 rows
  const bool head_x = decode && fam != ADEPT_FAMILY_BERT && m->dt == ADEPT_DTYPE_BF16 && head_rows_supported(D);
  m->xhead_ready = head_x;
  int32_t* exit_w = stop ? m->tok_exit : exit_out;
  launch_pass_init(st, n_tok, prompt_len, decode ? 1 : 0, m->tok_seq, m->tok_pos, m->row_tok[0], m->d_seq_len,
                   m->max_blocks_per_seq * c.kv_block_tokens, fam == ADEPT_FAMILY_LLAMA ? 0 : c.max_pos,
                   m->err_word, m->ctr, ctr_words(N), sim_out, N, stop ? m->tok_exit : nullptr);
  // passes of at most DG_MAX_M rows (bf16 decoders): the producer of each layer's input
  // (the embedding, then the exit kernel) also writes it standardised into xn, and the O
  // projection hands the tile statistics of its output to the FFN input's GEMM
  const bool dgrows = n_tok <= DG_MAX_M && m->dt == ADEPT_DTYPE_BF16 && m->use_dg && !m->force_simt &&
                      fam != ADEPT_FAMILY_BERT;
  launch_embed(st, m->dt, tokens, n_tok, m->tok_pos, m->tok_emb, m->pos_emb, m->type_emb, m->emb_g, m->emb_b, fam, D,
               m->V, eps, m->X_in[0], m->err_word, dgrows ? (bf16*)m->xn : nullptr, amode, eps);
  bool xn_valid = dgrows;   // xn holds X_in[par] standardised
  m->launches += 2;
  const KVCacheView cv = cache_view(m);
  const int causal = fam != ADEPT_FAMILY_BERT;
  // generation step: the split-KV attention grid covers the reserved capacity (CTAs past a
  // sequence's length return at once), which keeps every launch of a step step-invariant
  const int decode_keys = decode ? std::min(c.max_seq, m->max_blocks_per_seq * c.kv_block_tokens) : 0;
  // all-at-once exits apply to prompt passes (a generation step holds one token per sequence)
  const int aao_len = !decode && m->all_at_once ? prompt_len : 0;
  (void)batch;
  // generation steps of a few sequences: layer i's exit step is taken by layer i+1's QKV launch
  // (or, if that launch declines, launched on its own just before it)
  const bool fuse_exit = decode && dgrows && !cross && !stop && m->use_fused_exit && m->use_stream &&
                         n_tok <= DS_EXIT_MAX_ROWS && aao_len == 0;
  struct {
    bool on;
    int layer, par;
    float* Xi;
    float* Ii;
    int* rt;
  } pend = {false, 0, 0, nullptr, nullptr, nullptr};
  int par = 0;
  for (int i = 1; i <= N; ++i) {
    const int l0 = i - 1;
    const LayerW& w = m->L[l0];
    const DevRange act{nullptr, m->ctr + CTR_ACTIVE + par, 0};
    float* Xi = m->X_in[par];
    float* Ii = m->I[par];
    int* rt = m->row_tok[par];
    const int mr = n_tok;
    // QKV of the active rows, and (prefill) layer i's K/V of every token that exited
    // before layer i, from its mapped state (Sec. 4.3), in one grouped launch.
    GemmProblem pr[2];
    int mrs[2] = {mr, mr};
    memset(pr, 0, sizeof pr);
    pr[0].A = m->xn; pr[0].lda = D; pr[0].a_rows = n_tok; pr[0].B = w.w_qkv; pr[0].ldb = D; pr[0].rows = act;
    pr[0].N = Dq + 2 * Dkv; pr[0].K = D; pr[0].Bt = w.t_qkv; pr[0].bt_nkb = cdiv(D, TW_KB);
    pr[0].epi = epi_base();
    pr[0].epi.kind = EPI_QKV; pr[0].epi.bias = w.b_qkv; pr[0].epi.out_t = m->q; pr[0].epi.ld_t = Dq;
    pr[0].epi.row_tok = rt; pr[0].epi.tok_seq = m->tok_seq; pr[0].epi.tok_pos = m->tok_pos;
    pr[0].epi.cache = cv; pr[0].epi.layer0 = l0; pr[0].epi.n_q_cols = Dq; pr[0].epi.n_kv_cols = Dkv;
    pr[0].epi.head_dim = m->dh; pr[0].epi.rope = fam == ADEPT_FAMILY_LLAMA; pr[0].epi.rope_table = m->rope_table;
    // attention input: standardised (gain folded into W_qkv)
    if (!decode && i >= 3 && !stop) {
      pr[1] = kv_problem(m, l0, m->xfill, n_tok, DevRange{nullptr, m->ctr + CTR_EXITED, 0}, m->exit_tok, m->tok_seq,
                         m->tok_pos);
      launch_standardize(st, m->dt, Xi, D, nullptr, act, mr, D, amode, eps, m->xn, D);
      m->launches += 1;
      gemm(m, st, pr, 2, mrs, m->gemm_cls);
    } else {
      bool done = false;
      if (pend.on) {
        pend.on = false;
        const int pl = pend.layer, pp = pend.par;
        DsExit ex;
        ex.Xin = pend.Xi; ex.Xout = m->X_out; ex.I = pend.Ii; ex.Xnext = m->X_in[pp ^ 1]; ex.Inext = m->I[pp ^ 1];
        ex.hsm_s = m->hsm_s; ex.hsm_prev = m->hsm_prev; ex.hsm_I = m->hsm_I;
        ex.ctr = m->ctr; ex.row_tok = pend.rt; ex.row_tok_next = m->row_tok[pp ^ 1];
        ex.forced = forced; ex.delta = m->d_delta; ex.sim = sim_out; ex.exit_tok = m->exit_tok;
        ex.exit_layer = exit_w; ex.err = m->err_word;
        ex.par = pp; ex.layer = pl; ex.n_layers = N; ex.first = pl == 1; ex.test = pl >= 2;
        ex.metric = m->exit_metric; ex.norm_mode = amode; ex.eps = eps;
        done = streaming_gemm_exit(m, st, pr[0], mr, ex, m->gemm_cls) >= 0;
        if (done) {
          m->launches += 1;
        } else {
          // not taken: the exit step on its own first, then the product
          xn_valid = launch_exit_small(st, pend.Xi, m->X_out, pend.Ii, pl == 1, D, m->ctr, pp, pend.rt,
                                       m->row_tok[pp ^ 1], forced, pl, N, m->d_delta, pl >= 2, sim_out, m->exit_tok,
                                       exit_w, m->X_in[pp ^ 1], m->I[pp ^ 1], m->hsm_s, m->hsm_prev, m->hsm_I, mr,
                                       dgrows ? (bf16*)m->xn : nullptr, amode, eps, m->exit_metric, aao_len,
                                       m->tok_pos, m->err_word) &&
                     dgrows;
          m->launches += 1;
        }
      }
      if (!done) {
        if (xn_valid)
          gemm(m, st, pr, 1, mrs, m->gemm_cls);
        else
          gemm_std(m, st, pr[0], mr, Xi, D, nullptr, amode, eps, m->gemm_cls);
      }
    }
    // attention over every cached position of layer i
    {
      cudaEvent_t b = nullptr;
      prof_begin(m, ADEPT_PROF_ATTENTION, st, &b);
      launch_attention(st, m->dt, m->q, Dq, m->att, Dq, act, mr, rt, m->tok_seq, m->tok_pos, m->d_seq_len, cv, l0,
                       m->H, causal, decode_keys, m->attn_ws, m->attn_ctr, m->err_word, stop ? m->tok_exit : nullptr,
                       prompt_len, m->use_attn_tc ? m->T_max : 0, N);
      prof_end(m, ADEPT_PROF_ATTENTION, st, b, 0, 0);
      m->launches += 1;
    }
    // O projection + residual
    GemmProblem p;
    memset(&p, 0, sizeof p);
    p.a_rows = n_tok;   // the TMA view ends at this pass's rows: tiles past them read zeros, not memory
    p.A = m->att; p.lda = Dq; p.B = w.w_o; p.ldb = Dq; p.rows = act; p.N = D; p.K = Dq;
    p.Bt = w.t_o; p.bt_nkb = cdiv(Dq, TW_KB);
    p.epi = epi_base(); p.epi.kind = EPI_RESID; p.epi.bias = w.b_o; p.epi.out_f32 = m->X_out; p.epi.ld_f32 = D;
    p.epi.resid = Xi; p.epi.ld_resid = D;
    bool ts_valid = false;   // the O projection leaves the tile statistics of X_out for the FFN input
    if (dgrows) {
      p.epi.tile_stats = m->tile_stats;
      ts_valid = dg_takes(m, 1, p, mr, nullptr);
      if (!ts_valid) p.epi.tile_stats = nullptr;
    }
    gemm(m, st, &p, 1, &mr, m->gemm_cls);
    if (fam == ADEPT_FAMILY_BERT) {
      launch_layernorm_inplace(st, m->X_out, act, mr, D, w.ln1_g, w.ln1_b, eps);
      m->launches += 1;
    }
    if (cross) {
      // cross-attention sublayer (encoder-decoder decoders, Sec. 5.2): Q of LN_c(X_out) (gain
      // and shift folded into W_Qc), attention over all source positions of the token's
      // sequence (the source cache, not causal), W_Oc + residual into X_out
      GemmProblem pc;
      memset(&pc, 0, sizeof pc);
      pc.a_rows = n_tok;
      pc.A = m->xn; pc.lda = D; pc.B = w.w_cq; pc.ldb = D; pc.rows = act; pc.N = Dq; pc.K = D;
      pc.Bt = w.t_cq; pc.bt_nkb = cdiv(D, TW_KB);
      pc.epi = epi_base(); pc.epi.kind = EPI_ACT; pc.epi.act = ACT_NONE; pc.epi.bias = w.b_cq;
      pc.epi.out_t = m->q; pc.epi.ld_t = Dq;
      gemm_std(m, st, pc, mr, m->X_out, D, nullptr, amode, eps, m->gemm_cls, nullptr,
               ts_valid ? m->tile_stats : nullptr);
      {
        cudaEvent_t b = nullptr;
        prof_begin(m, ADEPT_PROF_ATTENTION, st, &b);
        launch_attention(st, m->dt, m->q, Dq, m->att, Dq, act, mr, rt, m->tok_seq, m->tok_pos, m->d_src_len,
                         cross_view(m), l0, m->H, 0, decode ? m->cs_blocks_per_seq * c.kv_block_tokens : 0,
                         m->attn_ws, m->attn_ctr, m->err_word, nullptr, 0, m->use_attn_tc ? m->T_max : 0, N);
        prof_end(m, ADEPT_PROF_ATTENTION, st, b, 0, 0);
        m->launches += 1;
      }
      pc.A = m->att; pc.lda = Dq; pc.B = w.w_co; pc.ldb = Dq; pc.N = D; pc.K = Dq;
      pc.Bt = w.t_co; pc.bt_nkb = cdiv(Dq, TW_KB);
      pc.epi = epi_base(); pc.epi.kind = EPI_RESID; pc.epi.bias = w.b_co; pc.epi.out_f32 = m->X_out;
      pc.epi.ld_f32 = D; pc.epi.resid = m->X_out; pc.epi.ld_resid = D;
      ts_valid = false;   // the statistics of the FFN input now come from this product
      if (dgrows) {
        pc.epi.tile_stats = m->tile_stats;
        ts_valid = dg_takes(m, 1, pc, mr, nullptr);
        if (!ts_valid) pc.epi.tile_stats = nullptr;
      }
      gemm(m, st, &pc, 1, &mr, m->gemm_cls);
    }
    // FFN (input standardised)
    p.A = m->xn; p.lda = D; p.B = w.w_up; p.ldb = D; p.N = w.up_rows; p.K = D;
    p.Bt = w.t_up; p.bt_nkb = cdiv(D, TW_KB);
    p.epi = epi_base();
    if (fam == ADEPT_FAMILY_LLAMA) {
      p.epi.kind = EPI_SWIGLU;
    } else {
      p.epi.kind = EPI_ACT;
      p.epi.act = fam == ADEPT_FAMILY_GPT2 ? ACT_GELU_TANH : ACT_GELU_ERF;
    }
    p.epi.bias = w.b_up; p.epi.out_t = m->hbuf; p.epi.ld_t = m->F;
    gemm_std(m, st, p, mr, m->X_out, D, nullptr, amode, eps, m->gemm_cls, nullptr, ts_valid ? m->tile_stats : nullptr);
    p.A = m->hbuf; p.lda = m->F; p.B = w.w_down; p.ldb = m->F; p.N = D; p.K = m->F;
    p.Bt = w.t_down; p.bt_nkb = cdiv(m->F, TW_KB);
    p.epi = epi_base(); p.epi.kind = EPI_RESID; p.epi.bias = w.b_down; p.epi.out_f32 = m->X_out; p.epi.ld_f32 = D;
    p.epi.resid = m->X_out; p.epi.ld_resid = D;
    gemm(m, st, &p, 1, &mr, m->gemm_cls);
    if (fam == ADEPT_FAMILY_BERT) {
      launch_layernorm_inplace(st, m->X_out, act, mr, D, w.ln2_g, w.ln2_b, eps);
      m->launches += 1;
    }
    if (i < N) {
      // exit test (Sec. 4.1) for 2 <= i <= N-1, inertia update, compaction (App. I)
      const int test = i >= 2;
      if (fuse_exit) {
        pend = {true, i, par, Xi, Ii, rt};
        xn_valid = false;
      } else if (n_tok <= EXIT_SMALL_MAX) {
        xn_valid = launch_exit_small(st, Xi, m->X_out, Ii, i == 1, D, m->ctr, par, rt, m->row_tok[par ^ 1], forced, i,
                                     N, m->d_delta, test, sim_out, m->exit_tok, exit_w, m->X_in[par ^ 1],
                                     m->I[par ^ 1], m->hsm_s, m->hsm_prev, m->hsm_I, mr,
                                     dgrows ? (bf16*)m->xn : nullptr, amode, eps, m->exit_metric, aao_len,
                                     m->tok_pos, m->err_word) &&
                   dgrows;
        m->launches += 1;
      } else {
        launch_exit_decide(st, m->X_out, Ii, Xi, D, act, mr, rt, forced, i, N, m->d_delta, test, m->exit_metric,
                           sim_out, m->flag, m->inv_norm, m->err_word);
        launch_exit_scan(st, m->ctr, par, m->flag, rt, m->row_tok[par ^ 1], m->exit_tok, m->dst, exit_w, i, aao_len,
                         m->tok_pos);
        launch_exit_move(st, Xi, m->X_out, Ii, i == 1, D, m->ctr + CTR_ACTIVE + par, mr, m->dst, m->inv_norm,
                         m->X_in[par ^ 1], m->I[par ^ 1], m->hsm_s, m->hsm_prev, m->hsm_I);
        m->launches += 3;
      }
      if (!decode && test) {
        // HSM of the tokens that left at layer i (Sec. 4.2); their s~_N feeds the fills
        run_hsm(m, st, DevRange{m->ctr + CTR_PREFIX + i - 1, m->ctr + CTR_PREFIX + i, 0}, mr, n_tok);
      }
      par ^= 1;
    } else {
      if (head_x)
        launch_final_scatter_head(st, m->X_out, D, m->ctr + CTR_ACTIVE + par, mr, rt, m->final_, exit_w, N,
                                  (bf16*)m->xhead, attn_norm_mode(m), m->cfg.norm_eps);
      else
        launch_final_scatter(st, m->X_out, D, m->ctr + CTR_ACTIVE + par, mr, rt, m->final_, exit_w, N);
      m->launches += 1;
    }
  }
  if (stop && exit_out)
    CUDA_TRY(m, cudaMemcpyAsync(exit_out, m->tok_exit, (size_t)n_tok * sizeof(int32_t), cudaMemcpyDeviceToDevice, st));
  if (decode && N >= 3) {
    // Generation step: the step's tokens belong to different sequences, so the HSM and
    // the skipped-layer fills of all exits run once, after the layer loop: one HSM over
    // every exited token, then one grouped launch over (skipped layer r) groups; rows are
    // in exit-layer order, so layer r's rows (i* < r) are a prefix.
    run_hsm(m, st, DevRange{nullptr, m->ctr + CTR_EXITED, 0}, n_tok, n_tok, head_x ? m->xhead : nullptr);
    std::vector<GemmProblem> probs;
    std::vector<int> mrs;
    for (int r = 3; r <= N; ++r) {
      probs.push_back(kv_problem(m, r - 1, m->xfill, n_tok, DevRange{nullptr, m->ctr + CTR_PREFIX + r - 1, 0}, m->exit_tok,
                                 m->tok_seq, m->tok_pos));
      mrs.push_back(n_tok);
    }
    // one weight-streaming launch over the skipped layers when the rows fit it, else the
    // grouped tcgen05 GEMM
    bool done = false;
    if (m->dt == ADEPT_DTYPE_BF16 && m->use_dg && !m->force_simt && n_tok <= DG_MAX_M) {
      cudaEvent_t b = nullptr;
      prof_begin(m, ADEPT_PROF_KV_FILL, st, &b);
      done = streaming_gemm_grouped(m, st, probs.data(), (int)probs.size(), n_tok) >= 0;
      prof_end(m, ADEPT_PROF_KV_FILL, st, b, 0, 0);
      if (done) m->launches += 1;
    }
    if (!done) gemm(m, st, probs.data(), (int)probs.size(), mrs.data(), ADEPT_PROF_KV_FILL);
  }
  return ADEPT_OK;
}

static adept_status run_head(adept_model* m, int batch, int prompt_len, bool decode, float* logits, int32_t* next,
                             cudaStream_t st) {
  const adept_config& c = m->cfg;
  const int D = m->D;
  const bool enc = c.family == ADEPT_FAMILY_BERT;
  float* out = logits ? logits : m->logits_ws;
  const bool rows_ready = !enc && decode && m->xhead_ready;   // head input already in xhead
  if (!rows_ready) {
    launch_head_rows(st, batch, decode ? 1 : prompt_len, enc ? 0 : 1, m->head_rows);
    m->launches += 1;
  }
  const DevRange rows{nullptr, nullptr, batch};
  GemmProblem p;
  memset(&p, 0, sizeof p);
  p.a_rows = batch;
  if (!enc) {
    p.A = m->xhead; p.lda = D; p.B = m->w_head; p.ldb = D; p.rows = rows; p.N = m->V; p.K = D;
    p.Bt = m->t_head; p.bt_nkb = cdiv(D, TW_KB);
    p.epi = epi_base(); p.epi.kind = EPI_F32; p.epi.bias = m->b_head; p.epi.out_f32 = out; p.epi.ld_f32 = m->V;
    if (rows_ready)
      gemm(m, st, &p, 1, &batch, m->gemm_cls);   // rows standardised by their producers
    else
      gemm_std(m, st, p, batch, m->final_, D, m->head_rows, attn_norm_mode(m), c.norm_eps, m->gemm_cls);
    if (next) m->launches += launch_argmax(st, out, m->V, batch, next, m->amax_v, m->amax_i);
  } else {
    p.A = m->xhead; p.lda = D; p.B = m->w_pool; p.ldb = D; p.rows = rows; p.N = D; p.K = D;
    p.epi = epi_base(); p.epi.kind = EPI_ACT; p.epi.act = ACT_TANH; p.epi.bias = m->b_pool; p.epi.out_t = m->pool_t;
    p.epi.ld_t = D;
    gemm_std(m, st, p, batch, m->final_, D, m->head_rows, NORM_COPY, c.norm_eps, m->gemm_cls);
    p.A = m->pool_t; p.lda = D; p.B = m->w_cls; p.ldb = D; p.N = c.n_classes; p.K = D;
    p.epi = epi_base(); p.epi.kind = EPI_F32; p.epi.bias = m->b_cls; p.epi.out_f32 = out; p.epi.ld_f32 = c.n_classes;
    gemm(m, st, &p, 1, &batch, m->gemm_cls);
    if (next) m->launches += launch_argmax(st, out, c.n_classes, batch, next, nullptr, nullptr);
  }
  return ADEPT_OK;
}

static adept_status check_launch(adept_model* m) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(m, ADEPT_ERR_CUDA, "kernel launch failed: %s", cudaGetErrorString(e));
  const adept_status d = m->deferred;
  m->deferred = ADEPT_OK;
  return d;   // the message was recorded where the error was met
}

// ---------------------------------------------------------------------------
// HSM training step (Sec. 4.2; Sec. 5.1 "Training"; App. D)
// ---------------------------------------------------------------------------

static void ht_free(adept_model* m) {
  if (!m->ht) return;
  for (void* p : m->ht->mine) {
    cudaFree(p);
    m->allocs.erase(std::remove(m->allocs.begin(), m->allocs.end(), p), m->allocs.end());
  }
  delete m->ht;
  m->ht = nullptr;
}

// C[M, N] (+)= A[M, K] B[N, K]^T (+ bias) into fp32 `out` (ld ldo); acc adds into out in place.
static GemmProblem ht_prob(const void* A, int lda, int a_rows, const void* B, int ldb, int M, int N, int K, float* out,
                           int ldo, const float* bias, bool acc) {
  GemmProblem p;
  memset(&p, 0, sizeof p);
  p.A = A; p.lda = lda; p.a_rows = a_rows; p.B = B; p.ldb = ldb;
  p.rows = DevRange{nullptr, nullptr, M}; p.N = N; p.K = K;
  p.epi = epi_base(); p.epi.kind = acc ? EPI_RESID : EPI_F32; p.epi.bias = bias;
  p.epi.out_f32 = out; p.epi.ld_f32 = ldo;
  if (acc) { p.epi.resid = out; p.epi.ld_resid = ldo; }
  return p;
}

// One launch over independent problems (a weight gradient and the matching input gradient
// share the launch, so that the small one does not leave SMs idle; K-split parts of one
// product likewise).
static void ht_gemm_n(adept_model* m, cudaStream_t st, const GemmProblem* ps, int n) {
  int mr[8];
  double fl = 0;
  for (int i = 0; i < n; ++i) {
    mr[i] = ps[i].rows.count;
    fl += 2.0 * ps[i].rows.count * ps[i].N * ps[i].K;
  }
  gemm(m, st, ps, n, mr, ADEPT_PROF_GEMM_TRAIN, fl, 0);
}

static void ht_gemm(adept_model* m, cudaStream_t st, std::initializer_list<GemmProblem> ps) {
  ht_gemm_n(m, st, ps.begin(), (int)ps.size());
}

constexpr int HT_DXH_SPLITS = 4;   // most K-splits of the head's input-gradient product

// K-splits of the head's input-gradient product (M = n, N = D, K = Vp): the count in 1..4 whose
// tiles (128 x 256) fill the SMs' last wave best, each split at least 512 of K.
static int ht_dxh_splits(int n, int D, int Vp, int sms) {
  const long long tiles = (long long)cdiv(n, 128) * cdiv(D, 256);
  int best = 1;
  double best_eff = 0;
  for (int s = 1; s <= HT_DXH_SPLITS; ++s) {
    if (s > 1 && Vp / s < 512) break;
    const double waves = (double)(tiles * s) / sms;
    const double eff = waves / std::ceil(waves);
    if (eff > best_eff + 1e-9) {
      best_eff = eff;
      best = s;
    }
  }
  return best;
}

static adept_status ht_init(adept_model* m, int cap, cudaStream_t st) {
  const adept_config& c = m->cfg;
  const int D = m->D, m1 = m->m1, m2 = m->m2, V = m->V, dt = m->dt;
  const size_t es = m->esz;
  ht_free(m);
  m->ht = new HsmTrain();
  HsmTrain& t = *m->ht;
  t.cap = cap;
  t.ldTc = (cap + 7) / 8 * 8;
  t.Vp = (V + 7) / 8 * 8;
  t.Vl = (V + 15) / 16 * 16;   // logits rows 64-byte aligned: the GEMM epilogue stores whole 16-float runs
  {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&t.sms, cudaDevAttrMultiProcessorCount, dev);
    t.sms = std::max(1, t.sms);
  }
  const long long n_el[HT_NPARAM] = {D, 9, 1, (long long)m1 * D, m1, (long long)m2 * m1, m2, (long long)m1 * m2,
                                     m1, m1, (long long)D * m1, D, D};
  long long o = 0;
  for (int i = 0; i < HT_NPARAM; ++i) {
    if (i != HT_CONV_B) o = (o + 15) / 16 * 16;
    t.off[i] = o;
    t.numel[i] = n_el[i];
    o += n_el[i];
  }
  t.off[HT_NPARAM] = (o + 15) / 16 * 16;
  const size_t P = (size_t)t.off[HT_NPARAM];
  auto A = [&](auto** p, size_t bytes) -> adept_status {
    TRY(dalloc(m, (void**)p, bytes));
    t.mine.push_back((void*)*p);
    return ADEPT_OK;
  };
  const size_t n = cap, L = t.ldTc;
  const bool enc = c.family == ADEPT_FAMILY_BERT;
  TRY(A(&t.theta, P * 4)); TRY(A(&t.grad, P * 4)); TRY(A(&t.mom1, P * 4)); TRY(A(&t.mom2, P * 4));
  TRY(A(&t.w1T, (size_t)m1 * D * es)); TRY(A(&t.w2T, (size_t)m2 * m1 * es));
  TRY(A(&t.w3T, (size_t)m1 * m2 * es)); TRY(A(&t.w4T, (size_t)D * m1 * es));
  if (enc) {
    TRY(A(&t.poolT, (size_t)D * D * es)); TRY(A(&t.zp, n * D * 4)); TRY(A(&t.dpt, n * D * es));
    TRY(A(&t.lossc, n * 4));
  } else {
    TRY(A(&t.headT, (size_t)D * t.Vp * es));
  }
  TRY(A(&t.iota, n * 4));
  TRY(A(&t.c0f, n * D * 4)); TRY(A(&t.z1f, n * m1 * 4)); TRY(A(&t.h1f, n * m1 * 4)); TRY(A(&t.z2f, n * m2 * 4));
  TRY(A(&t.h3f, n * m1 * 4)); TRY(A(&t.h5f, n * D * 4)); TRY(A(&t.stf, n * D * 4));
  if (!enc) TRY(A(&t.logits, n * t.Vl * 4));
  TRY(A(&t.lossr, n * 4)); TRY(A(&t.dxh, (size_t)HT_DXH_SPLITS * n * D * 4)); TRY(A(&t.dc0f, n * D * 4)); TRY(A(&t.dh5f, n * D * 4));
  TRY(A(&t.dh4f, n * m1 * 4)); TRY(A(&t.dh3f, n * m1 * 4)); TRY(A(&t.dh2f, n * m2 * 4));
  TRY(A(&t.r1, n * 4)); TRY(A(&t.r2, n * 4)); TRY(A(&t.cw, n * 10 * 4));
  t.part_cols = std::max({2 * D, 2 * m1, m2, D + 10});
  TRY(A(&t.part, (size_t)ht_colsum_chunks(cap) * t.part_cols * 4));
  TRY(A(&t.c0t, n * D * es)); TRY(A(&t.c0T, (size_t)D * L * es));
  TRY(A(&t.h1t, n * m1 * es)); TRY(A(&t.h1T, (size_t)m1 * L * es));
  TRY(A(&t.h2t, n * m2 * es)); TRY(A(&t.h2T, (size_t)m2 * L * es));
  TRY(A(&t.h4t, n * m1 * es)); TRY(A(&t.h4T, (size_t)m1 * L * es));
  TRY(A(&t.xht, n * D * es));
  if (!enc) TRY(A(&t.dlt, n * t.Vp * es));
  TRY(A(&t.dh5t, n * D * es)); TRY(A(&t.dh5T, (size_t)D * L * es));
  TRY(A(&t.dh3t, n * m1 * es)); TRY(A(&t.dh3T, (size_t)m1 * L * es));
  TRY(A(&t.dz2t, n * m2 * es)); TRY(A(&t.dz2T, (size_t)m2 * L * es));
  if (dt != ADEPT_DTYPE_BF16 || m->force_simt) {
    // SIMT GEMMs stage C in the model's scratch: size it for the largest training product now
    const size_t big = std::max({n * (size_t)std::max({enc ? D : V, m2, m1, D}), (size_t)m1 * m2, (size_t)m1 * D});
    if (!ensure_scratch(m, big)) return ADEPT_ERR_OOM;
  }
  // master parameters = the model's HSM weights; zero gradients and moments
  CUDA_TRY(m, cudaMemsetAsync(t.theta, 0, P * 4, st));
  CUDA_TRY(m, cudaMemsetAsync(t.grad, 0, P * 4, st));
  CUDA_TRY(m, cudaMemsetAsync(t.mom1, 0, P * 4, st));
  CUDA_TRY(m, cudaMemsetAsync(t.mom2, 0, P * 4, st));
  const std::pair<int, const float*> vecs[] = {{HT_G0, m->hsm_g0}, {HT_FC1_B, m->hsm_b1}, {HT_FC2_B, m->hsm_b2},
                                               {HT_FC3_B, m->hsm_b3}, {HT_G1, m->hsm_g1}, {HT_FC4_B, m->hsm_b4},
                                               {HT_G2, m->hsm_g2}};
  for (const auto& v : vecs)
    CUDA_TRY(m, cudaMemcpyAsync(t.theta + t.off[v.first], v.second, t.numel[v.first] * 4, cudaMemcpyDeviceToDevice, st));
  CUDA_TRY(m, cudaMemcpyAsync(t.theta + t.off[HT_CONV_W], m->hsm_conv, 10 * 4, cudaMemcpyDeviceToDevice, st));
  launch_to_f32(st, dt, m->hsm_w1, t.theta + t.off[HT_FC1_W], (int)t.numel[HT_FC1_W]);
  launch_to_f32(st, dt, m->hsm_w2, t.theta + t.off[HT_FC2_W], (int)t.numel[HT_FC2_W]);
  launch_to_f32(st, dt, m->hsm_w3, t.theta + t.off[HT_FC3_W], (int)t.numel[HT_FC3_W]);
  launch_to_f32(st, dt, m->hsm_w4, t.theta + t.off[HT_FC4_W], (int)t.numel[HT_FC4_W]);
  // transposed copies: W1^T [D][m1], W2^T [m1][m2], W3^T [m2][m1], W4^T [m1][D], head^T [D][Vp]
  ht_launch_transpose(st, dt, m->hsm_w1, m1, D, t.w1T, m1);
  ht_launch_transpose(st, dt, m->hsm_w2, m2, m1, t.w2T, m2);
  ht_launch_transpose(st, dt, m->hsm_w3, m1, m2, t.w3T, m1);
  ht_launch_transpose(st, dt, m->hsm_w4, D, m1, t.w4T, D);
  if (enc) ht_launch_transpose(st, dt, m->w_pool, D, D, t.poolT, D);
  else ht_launch_transpose(st, dt, m->w_head, V, D, t.headT, t.Vp);
  std::vector<int> io(cap);
  for (int i = 0; i < cap; ++i) io[i] = i;
  CUDA_TRY(m, cudaMemcpyAsync(t.iota, io.data(), (size_t)cap * 4, cudaMemcpyHostToDevice, st));
  CUDA_TRY(m, cudaStreamSynchronize(st));
  return check_launch(m);
}

// Table S1 forward on n rows, keeping what the backward reads; the mapped state s~ lands in
// stf (fp32) and, standardised for the head (decoders) or as it is (encoders), in xht (T).
static void ht_forward(adept_model* m, cudaStream_t st, int n, const float* s_i, const float* s_prev,
                       const float* inertia) {
  HsmTrain& t = *m->ht;
  const int D = m->D, m1 = m->m1, m2 = m->m2, dt = m->dt;
  const int ldT = (n + 7) / 8 * 8;
  const float eps = m->cfg.hsm_eps, neps = m->cfg.norm_eps;
  const int hmode = attn_norm_mode(m);
  const DevRange rows{nullptr, nullptr, n};
  auto P = [&](int i) { return t.theta + t.off[i]; };
  launch_hsm_prep(st, dt, s_i, s_prev, inertia, rows, n, D, P(HT_G0), P(HT_CONV_W), eps, t.c0f, t.c0t);
  ht_gemm(m, st, {ht_prob(t.c0t, D, n, m->hsm_w1, D, n, m1, D, t.z1f, m1, P(HT_FC1_B), false)});
  ht_launch_gelu_tile(st, dt, 0, t.z1f, t.h1f, n, m1, t.h1t, t.h1T, ldT, nullptr);
  ht_gemm(m, st, {ht_prob(t.h1t, m1, n, m->hsm_w2, m1, n, m2, m1, t.z2f, m2, P(HT_FC2_B), false)});
  ht_launch_gelu_tile(st, dt, 0, t.z2f, nullptr, n, m2, t.h2t, t.h2T, ldT, nullptr);
  ht_gemm(m, st, {ht_prob(t.h2t, m2, n, m->hsm_w3, m2, n, m1, m2, t.h3f, m1, P(HT_FC3_B), false)});
  launch_hsm_mid(st, dt, t.h3f, t.h1f, rows, n, m1, P(HT_G1), eps, t.h4t);
  ht_gemm(m, st, {ht_prob(t.h4t, m1, n, m->hsm_w4, m1, n, D, m1, t.h5f, D, P(HT_FC4_B), false)});
  launch_hsm_out(st, dt, t.h5f, t.c0f, nullptr, 0, rows, n, D, P(HT_G2), eps, t.iota, t.stf, t.xht, hmode, neps);
}

// Backward of Table S1 from dxh (nsplit partial sums [n][D] of the gradient with respect to
// the head's input), then AdamW and the write-back of the model's HSM weights.  `launches`:
// the caller's own non-GEMM launches, added to the count.
static adept_status ht_backward(adept_model* m, cudaStream_t st, int n, int nsplit, const float* s_i,
                                const float* s_prev, const float* inertia, const adept_adamw& hp, int launches) {
  HsmTrain& t = *m->ht;
  const int D = m->D, m1 = m->m1, m2 = m->m2, dt = m->dt;
  const int ldT = (n + 7) / 8 * 8;
  const float eps = m->cfg.hsm_eps, neps = m->cfg.norm_eps;
  const int hmode = attn_norm_mode(m);
  auto P = [&](int i) { return t.theta + t.off[i]; };
  auto G = [&](int i) { return t.grad + t.off[i]; };
  ht_launch_out_bwd(st, dt, t.dxh, nsplit, (size_t)n * D, t.stf, t.h5f, n, D, P(HT_G2), eps, hmode, neps, t.dc0f,
                    t.dh5f, t.dh5t, t.r2);
  int cl = 0;
  {
    ColJobs J{};
    J.n = n; J.nj = 2;
    J.j[0] = ColJob{t.dh5f, nullptr, nullptr, D, G(HT_FC4_B)};
    J.j[1] = ColJob{t.dc0f, t.h5f, t.r2, D, G(HT_G2)};
    cl += ht_launch_colsum(st, J, t.part);
  }
  ht_launch_transpose(st, dt, t.dh5t, n, D, t.dh5T, ldT);
  ht_launch_transpose(st, dt, t.h4t, n, m1, t.h4T, ldT);
  ht_gemm(m, st, {ht_prob(t.dh5T, ldT, D, t.h4T, ldT, D, m1, ldT, G(HT_FC4_W), m1, nullptr, false),    // dW4
                   ht_prob(t.dh5t, D, n, t.w4T, D, n, m1, D, t.dh4f, m1, nullptr, false)});            // dh4
  ht_launch_mid_bwd(st, dt, t.dh4f, t.h3f, n, m1, P(HT_G1), eps, t.dh3f, t.dh3t, t.r1);
  {
    ColJobs J{};
    J.n = n; J.nj = 2;
    J.j[0] = ColJob{t.dh4f, t.h3f, t.r1, m1, G(HT_G1)};
    J.j[1] = ColJob{t.dh3f, nullptr, nullptr, m1, G(HT_FC3_B)};
    cl += ht_launch_colsum(st, J, t.part);
  }
  ht_launch_transpose(st, dt, t.dh3t, n, m1, t.dh3T, ldT);
  ht_gemm(m, st, {ht_prob(t.dh3T, ldT, m1, t.h2T, ldT, m1, m2, ldT, G(HT_FC3_W), m2, nullptr, false),   // dW3
                   ht_prob(t.dh3t, m1, n, t.w3T, m1, n, m2, m1, t.dh2f, m2, nullptr, false)});          // dh2
  ht_launch_gelu_tile(st, dt, 1, t.z2f, t.dh2f, n, m2, t.dz2t, t.dz2T, ldT, t.part);
  {
    ColJobs J{};
    J.n = n; J.nj = 1;
    J.j[0] = ColJob{nullptr, nullptr, nullptr, m2, G(HT_FC2_B)};
    cl += ht_launch_colsum_finish(st, J, t.part);
  }
  ht_gemm(m, st, {ht_prob(t.dz2T, ldT, m2, t.h1T, ldT, m2, m1, ldT, G(HT_FC2_W), m1, nullptr, false),   // dW2
                   ht_prob(t.dz2t, m2, n, t.w2T, m2, n, m1, m2, t.dh4f, m1, nullptr, true)});           // dh1 = dh4 + dz2 W2
  ht_launch_gelu_tile(st, dt, 1, t.z1f, t.dh4f, n, m1, t.dh3t, t.dh3T, ldT, t.part);  // dz1 (dh3's buffers are free)
  {
    ColJobs J{};
    J.n = n; J.nj = 1;
    J.j[0] = ColJob{nullptr, nullptr, nullptr, m1, G(HT_FC1_B)};
    cl += ht_launch_colsum_finish(st, J, t.part);
  }
  ht_launch_transpose(st, dt, t.c0t, n, D, t.c0T, ldT);
  ht_gemm(m, st, {ht_prob(t.dh3T, ldT, m1, t.c0T, ldT, m1, D, ldT, G(HT_FC1_W), D, nullptr, false),    // dW1
                   ht_prob(t.dh3t, m1, n, t.w1T, m1, n, D, m1, t.dc0f, D, nullptr, true)});             // dc0 += dz1 W1
  ht_launch_prep_bwd(st, s_i, s_prev, inertia, t.dc0f, n, D, P(HT_G0), P(HT_CONV_W), eps, t.dh5f, t.cw);
  {
    ColJobs J{};
    J.n = n; J.nj = 2;
    J.j[0] = ColJob{t.dh5f, nullptr, nullptr, D, G(HT_G0)};
    J.j[1] = ColJob{t.cw, nullptr, nullptr, 10, G(HT_CONV_W)};
    cl += ht_launch_colsum(st, J, t.part);
  }
  // AdamW, writing the updated values back into the model's HSM weights
  t.step += 1;
  AdamArgs a{};
  a.theta = t.theta; a.grad = t.grad; a.m = t.mom1; a.v = t.mom2;
  a.lr = hp.lr; a.b1 = hp.beta1; a.b2 = hp.beta2; a.eps = hp.eps; a.wd = hp.weight_decay;
  a.ibc1 = (float)(1.0 / (1.0 - std::pow((double)hp.beta1, (double)t.step)));
  a.ibc2 = (float)(1.0 / (1.0 - std::pow((double)hp.beta2, (double)t.step)));
  const AdamSeg segs[] = {
      {t.off[HT_G0], 1, D, m->hsm_g0, nullptr, nullptr, 0, 0},
      {t.off[HT_CONV_W], 1, 10, m->hsm_conv, nullptr, nullptr, 0, 0},
      {t.off[HT_FC1_W], m1, D, nullptr, m->hsm_w1, t.w1T, 0, 0},
      {t.off[HT_FC1_B], 1, m1, m->hsm_b1, nullptr, nullptr, 0, 0},
      {t.off[HT_FC2_W], m2, m1, nullptr, m->hsm_w2, t.w2T, 0, 0},
      {t.off[HT_FC2_B], 1, m2, m->hsm_b2, nullptr, nullptr, 0, 0},
      {t.off[HT_FC3_W], m1, m2, nullptr, m->hsm_w3, t.w3T, 0, 0},
      {t.off[HT_FC3_B], 1, m1, m->hsm_b3, nullptr, nullptr, 0, 0},
      {t.off[HT_G1], 1, m1, m->hsm_g1, nullptr, nullptr, 0, 0},
      {t.off[HT_FC4_W], D, m1, nullptr, m->hsm_w4, t.w4T, 0, 0},
      {t.off[HT_FC4_B], 1, D, m->hsm_b4, nullptr, nullptr, 0, 0},
      {t.off[HT_G2], 1, D, m->hsm_g2, nullptr, nullptr, 0, 0}};
  a.nseg = (int)(sizeof segs / sizeof segs[0]);
  for (int i = 0; i < a.nseg; ++i) a.seg[i] = segs[i];
  ht_launch_adamw(st, dt, a);
  TRY(retile_hsm(m, st, false));   // the generation steps' copies follow the updated weights
  // launches outside ht_gemm: prep, 2 GELU, mid, out (forward), out_bwd, mid_bwd, 2 GELU', prep_bwd,
  // 4 transposes, the column sums and AdamW, and the caller's loss launches
  m->launches += 15 + launches + cl;
  return check_launch(m);
}

// Decoder step (Sec. 4.2): the frozen head (final-norm gain and shift folded into its
// weights), next-token cross-entropy, and the head's input gradient dxh = dlogits W_head with
// K = Vp split into parts that the backward's first kernel sums.
static adept_status ht_step(adept_model* m, int n, const float* s_i, const float* s_prev, const float* inertia,
                            const int32_t* target, const adept_adamw& hp, float* loss, cudaStream_t st) {
  HsmTrain& t = *m->ht;
  const int D = m->D, V = m->V, Vp = t.Vp, dt = m->dt;
  ht_forward(m, st, n, s_i, s_prev, inertia);
  ht_gemm(m, st, {ht_prob(t.xht, D, n, m->w_head, D, n, V, D, t.logits, t.Vl, m->b_head, false)});
  ht_launch_ce(st, dt, t.logits, t.Vl, n, V, Vp, target, t.lossr, t.dlt, loss, m->err_word);
  const int S0 = ht_dxh_splits(n, D, Vp, t.sms);
  const int kc = (cdiv(Vp, S0) + 63) / 64 * 64;
  GemmProblem ps[HT_DXH_SPLITS];
  int S = 0;
  for (int k0 = 0; k0 < Vp; k0 += kc, ++S)
    ps[S] = ht_prob((const char*)t.dlt + (size_t)k0 * m->esz, Vp, n, (const char*)t.headT + (size_t)k0 * m->esz, Vp, n,
                    D, std::min(kc, Vp - k0), t.dxh + (size_t)S * n * D, D, nullptr, false);
  ht_gemm_n(m, st, ps, S);
  return ht_backward(m, st, n, S, s_i, s_prev, inertia, hp, 1 + (loss ? 1 : 0));
}

// Encoder step (Sec. 4.3): similarity rows against the original final states, then, on the
// first n_cls rows, the frozen pooler (dense + tanh) and classifier with their cross-entropy;
// the pooler's input gradient adds into those rows of dxh.
static adept_status ht_step_cls(adept_model* m, int n, const float* s_i, const float* s_prev, const float* inertia,
                                const float* s_final, int n_cls, const int32_t* label, float cls_weight,
                                const adept_adamw& hp, float* loss, cudaStream_t st) {
  HsmTrain& t = *m->ht;
  const int D = m->D, dt = m->dt;
  ht_forward(m, st, n, s_i, s_prev, inertia);
  ht_launch_cos(st, t.stf, s_final, n, D, t.lossr, t.dxh);
  int own = 1;
  const float wc = n_cls > 0 ? cls_weight / (float)n_cls : 0.f;
  if (n_cls > 0) {
    ht_gemm(m, st, {ht_prob(t.xht, D, n_cls, m->w_pool, D, n_cls, D, D, t.zp, D, m->b_pool, false)});
    ht_launch_cls(st, dt, t.zp, n_cls, D, m->w_cls, m->b_cls, m->cfg.n_classes, label, wc, t.lossc, t.dpt, m->err_word);
    ht_gemm(m, st, {ht_prob(t.dpt, D, n_cls, t.poolT, D, n_cls, D, D, t.dxh, D, nullptr, true)});
    ++own;
  }
  if (loss) {
    ht_launch_loss(st, t.lossr, n, 1.f / (float)n, t.lossc, n_cls, wc, loss);
    ++own;
  }
  return ht_backward(m, st, n, 1, s_i, s_prev, inertia, hp, own);
}

static bool adamw_ok(const adept_adamw* hp) {
  return hp->lr >= 0.f && hp->beta1 >= 0.f && hp->beta1 < 1.f && hp->beta2 >= 0.f && hp->beta2 < 1.f && hp->eps > 0.f &&
         hp->weight_decay >= 0.f;
}


// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" {

const char* adept_status_string(adept_status s) {
  switch (s) {
    case ADEPT_OK: return "ok";
    case ADEPT_ERR_INVALID_ARG: return "invalid argument";
    case ADEPT_ERR_OOM: return "out of device memory";
    case ADEPT_ERR_CAPACITY: return "capacity exceeded";
    case ADEPT_ERR_CUDA: return "CUDA error";
    case ADEPT_ERR_TIMEOUT: return "device wait timed out";
    case ADEPT_ERR_DEVICE_INPUT: return "invalid device-side input";
  }
  return "unknown status";
}

const char* adept_last_error(const adept_model* m) { return m ? m->err.c_str() : g_load_error.c_str(); }

adept_status adept_model_load(const adept_config* cfg_in, const adept_tensor_table* weights, void* stream,
                              adept_model** out) {
  g_load_error.clear();
  if (!cfg_in || !weights || !out) return fail(nullptr, ADEPT_ERR_INVALID_ARG, "NULL argument");
  *out = nullptr;
  adept_config cfg = *cfg_in;
  TRY(validate_cfg(&cfg));
  if (weights->n_tensors < 0 || (weights->n_tensors > 0 && !weights->tensors))
    return fail(nullptr, ADEPT_ERR_INVALID_ARG, "bad tensor table");
  adept_model* m = new adept_model();
  m->cfg = cfg;
  m->N = cfg.n_layers; m->D = cfg.d_model; m->H = cfg.n_heads; m->Hkv = cfg.n_kv_heads; m->dh = cfg.head_dim;
  m->Dq = m->H * m->dh; m->Dkv = m->Hkv * m->dh; m->F = cfg.d_ffn; m->V = cfg.vocab;
  m->m1 = cfg.hsm_m1; m->m2 = cfg.hsm_m2; m->dt = cfg.dtype; m->esz = cfg.dtype == ADEPT_DTYPE_BF16 ? 2 : 4;
  m->T_max = cfg.max_pass_tokens > 0 ? cfg.max_pass_tokens : cfg.max_batch * cfg.max_seq;
  if (m->T_max < cfg.max_batch) m->T_max = cfg.max_batch;
  Loader ld;
  ld.m = m;
  ld.st = (cudaStream_t)stream;
  for (int i = 0; i < weights->n_tensors; ++i) {
    const adept_tensor& t = weights->tensors[i];
    if (!t.name) {
      free_all(m);
      delete m;
      return fail(nullptr, ADEPT_ERR_INVALID_ARG, "tensor %d has no name", i);
    }
    ld.t[t.name] = t;
  }
  adept_status s = load_weights(m, ld);
  if (s == ADEPT_OK) s = alloc_runtime(m);
  if (s == ADEPT_OK) s = make_tiled(m, ld.st);
  if (s == ADEPT_OK) {
    cudaError_t e = cudaStreamSynchronize(ld.st);
    if (e != cudaSuccess) s = fail(m, ADEPT_ERR_CUDA, "load: %s", cudaGetErrorString(e));
  }
  if (s != ADEPT_OK) {
    g_load_error = m->err;
    free_all(m);
    delete m;
    return s;
  }
  // the staging buffers are not needed after loading
  for (auto it = m->allocs.begin(); it != m->allocs.end();) {
    if (*it == ld.staging || *it == ld.fstage[0] || *it == ld.fstage[1]) {
      cudaFree(*it);
      it = m->allocs.erase(it);
    } else {
      ++it;
    }
  }
  *out = m;
  return ADEPT_OK;
}

void adept_free(adept_model* m) {
  if (!m) return;
  cudaDeviceSynchronize();
  free_all(m);
  delete m;
}

static adept_status check_cross_set(adept_model* m, int batch) {
  if (m->cfg.max_src <= 0) return ADEPT_OK;
  for (int b = 0; b < batch; ++b)
    if (m->h_src_len[b] <= 0)
      return fail(m, ADEPT_ERR_INVALID_ARG, "sequence %d has no cross-attention source (adept_set_cross_source)", b);
  return ADEPT_OK;
}

adept_status adept_prefill(adept_model* m, int batch, int prompt_len, const int32_t* d_tokens, float delta,
                           const int32_t* d_forced_exit, int32_t* d_exit_layer_out, float* d_logits_out,
                           int32_t* d_next_token_out, float* d_sim_out, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (!d_tokens) return fail(m, ADEPT_ERR_INVALID_ARG, "d_tokens is NULL");
  if (batch < 1 || prompt_len < 1) return fail(m, ADEPT_ERR_INVALID_ARG, "batch and prompt_len must be positive");
  if (batch > m->cfg.max_batch) return fail(m, ADEPT_ERR_CAPACITY, "batch %d > max_batch %d", batch, m->cfg.max_batch);
  if (prompt_len > m->cfg.max_seq)
    return fail(m, ADEPT_ERR_CAPACITY, "prompt_len %d > max_seq %d", prompt_len, m->cfg.max_seq);
  if (std::isnan(delta)) return fail(m, ADEPT_ERR_INVALID_ARG, "delta is NaN");
  if ((long long)batch * prompt_len > m->T_max)
    return fail(m, ADEPT_ERR_CAPACITY, "batch * prompt_len %d above the pass workspace (%d rows)", batch * prompt_len,
                m->T_max);
  TRY(check_cross_set(m, batch));
  cudaStream_t st = (cudaStream_t)stream;
  std::vector<int> lens(batch, prompt_len);
  TRY(reserve_seqs(m, batch, lens.data(), st));
  launch_set_float(st, m->d_delta, delta);
  m->launches += 1;
  TRY(run_pass(m, batch * prompt_len, batch, prompt_len, false, d_tokens, d_forced_exit, d_exit_layer_out, d_sim_out,
               st));
  TRY(run_head(m, batch, prompt_len, false, d_logits_out, d_next_token_out, st));
  span_collect(m, st);
  return check_launch(m);
}

adept_status adept_set_cross_source(adept_model* m, int n_seq, const int32_t* h_src_len, const float* d_states,
                                    void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  const adept_config& c = m->cfg;
  if (c.max_src <= 0) return fail(m, ADEPT_ERR_INVALID_ARG, "the model has no cross-attention (max_src = 0)");
  if (!h_src_len || !d_states) return fail(m, ADEPT_ERR_INVALID_ARG, "NULL source lengths or states");
  if (n_seq < 1 || n_seq > c.max_batch) return fail(m, ADEPT_ERR_INVALID_ARG, "n_seq %d out of range", n_seq);
  std::vector<int> seq, pos;
  for (int b = 0; b < n_seq; ++b) {
    if (h_src_len[b] < 1 || h_src_len[b] > c.max_src)
      return fail(m, ADEPT_ERR_INVALID_ARG, "source length %d of sequence %d outside [1, %d]", h_src_len[b], b, c.max_src);
    for (int p = 0; p < h_src_len[b]; ++p) {
      seq.push_back(b);
      pos.push_back(p);
    }
  }
  PdlScope pdl(!m->profile);
  cudaStream_t st = (cudaStream_t)stream;
  const int n = (int)seq.size(), D = m->D;
  CUDA_TRY(m, cudaMemcpyAsync(m->cs_seq, seq.data(), n * sizeof(int), cudaMemcpyHostToDevice, st));
  CUDA_TRY(m, cudaMemcpyAsync(m->cs_pos, pos.data(), n * sizeof(int), cudaMemcpyHostToDevice, st));
  // the states in the GEMM input type, then every layer's source K/V in one grouped launch
  launch_standardize(st, m->dt, d_states, D, nullptr, DevRange{nullptr, nullptr, n}, n, D, NORM_COPY, 0.f, m->cs_x, D);
  m->launches += 1;
  std::vector<GemmProblem> probs(m->N);
  std::vector<int> mrs(m->N, n);
  const KVCacheView cv = cross_view(m);
  for (int l = 0; l < m->N; ++l) {
    GemmProblem& p = probs[l];
    memset(&p, 0, sizeof p);
    p.A = m->cs_x; p.lda = D; p.a_rows = n;
    p.B = m->L[l].w_ckv; p.ldb = D; p.N = 2 * m->Dkv; p.K = D;
    p.rows = DevRange{nullptr, nullptr, n};
    p.epi = epi_base();
    p.epi.kind = EPI_KV; p.epi.bias = m->L[l].b_ckv;
    p.epi.row_tok = m->cs_iota; p.epi.tok_seq = m->cs_seq; p.epi.tok_pos = m->cs_pos;
    p.epi.cache = cv; p.epi.layer0 = l;
    p.epi.n_q_cols = 0; p.epi.n_kv_cols = m->Dkv; p.epi.head_dim = m->dh;
  }
  gemm(m, st, probs.data(), m->N, mrs.data(), ADEPT_PROF_GEMM_PREFILL);
  // the lengths last: a copy on the stream starts after the projection has completed, so no
  // later kernel's early (pre-dependency-wait) reads of the source cache can overlap it
  for (int b = 0; b < n_seq; ++b) m->h_src_len[b] = h_src_len[b];
  CUDA_TRY(m, cudaMemcpyAsync(m->d_src_len, m->h_src_len.data(), n_seq * sizeof(int), cudaMemcpyHostToDevice, st));
  CUDA_TRY(m, cudaStreamSynchronize(st));   // the host vectors above are released on return
  return check_launch(m);
}

adept_status adept_decode_step(adept_model* m, int batch, const int32_t* d_tokens, float delta,
                               const int32_t* d_forced_exit, int32_t* d_exit_layer_out, float* d_logits_out,
                               int32_t* d_next_token_out, float* d_sim_out, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (m->cfg.family == ADEPT_FAMILY_BERT) return fail(m, ADEPT_ERR_INVALID_ARG, "decode needs a decoder model");
  if (!d_tokens) return fail(m, ADEPT_ERR_INVALID_ARG, "d_tokens is NULL");
  if (batch < 1 || batch > m->cfg.max_batch) return fail(m, ADEPT_ERR_CAPACITY, "batch %d out of range", batch);
  if (std::isnan(delta)) return fail(m, ADEPT_ERR_INVALID_ARG, "delta is NaN");
  TRY(check_cross_set(m, batch));
  for (int b = 0; b < batch; ++b) {
    if (m->seq_blocks[b].empty()) return fail(m, ADEPT_ERR_INVALID_ARG, "sequence %d has no prompt", b);
    if (m->h_seq_len[b] >= m->max_blocks_per_seq * m->cfg.kv_block_tokens || m->h_seq_len[b] >= m->cfg.max_seq)
      return fail(m, ADEPT_ERR_CAPACITY, "sequence %d is full (%d positions)", b, m->h_seq_len[b]);
  }
  cudaStream_t st = (cudaStream_t)stream;
  // inputs into the staging buffers; the step itself reads and writes only those
  launch_stage_in(st, m->d_delta, delta, d_tokens, m->dec_tok, d_forced_exit, m->dec_forced, batch);
  m->launches += 1;
  auto body = [&](cudaStream_t s) -> adept_status {
    TRY(run_pass(m, batch, batch, 1, true, m->dec_tok, m->dec_forced, m->dec_exit, m->dec_sim, s));
    TRY(run_head(m, batch, 1, true, m->logits_ws, m->dec_next, s));
    span_collect(m, s);
    return ADEPT_OK;
  };
  const bool graph_ok = m->use_graph && !m->profile;
  if (graph_ok && m->dec_warm[batch] >= 1) {
    if (!m->dec_graph[batch]) {
      // capture one generation step on a private stream; later steps replay it
      if (!m->cap_stream) CUDA_TRY(m, cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking));
      const int64_t l0 = m->launches;
      CUDA_TRY(m, cudaStreamBeginCapture(m->cap_stream, cudaStreamCaptureModeThreadLocal));
      adept_status s = body(m->cap_stream);
      cudaGraph_t g = nullptr;
      cudaError_t e = cudaStreamEndCapture(m->cap_stream, &g);
      if (s != ADEPT_OK) {
        if (g) cudaGraphDestroy(g);
        return s;
      }
      if (e != cudaSuccess) return fail(m, ADEPT_ERR_CUDA, "graph capture failed: %s", cudaGetErrorString(e));
      cudaGraphExec_t ex = nullptr;
      e = cudaGraphInstantiate(&ex, g, 0);
      cudaGraphDestroy(g);
      if (e != cudaSuccess) return fail(m, ADEPT_ERR_CUDA, "graph instantiate failed: %s", cudaGetErrorString(e));
      m->dec_graph[batch] = ex;
      m->graph_launches = m->launches - l0;
      m->launches = l0;
    }
    CUDA_TRY(m, cudaGraphLaunch(m->dec_graph[batch], st));
    m->launches += m->graph_launches;
  } else {
    TRY(body(st));
    m->dec_warm[batch] += 1;
  }
  for (int b = 0; b < batch; ++b) m->h_seq_len[b] += 1;
  // outputs out of the staging buffers, one launch
  if (d_exit_layer_out || d_next_token_out || d_logits_out || d_sim_out) {
    launch_stage_out(st, batch, m->dec_exit, d_exit_layer_out, m->dec_next, d_next_token_out, m->logits_ws,
                     d_logits_out, (long long)batch * m->V, m->dec_sim, d_sim_out, batch * m->N);
    m->launches += 1;
  }
  return check_launch(m);
}

adept_status adept_calibrate_threshold(adept_model* m, int batch, int prompt_len, const int32_t* d_tokens,
                                       float target_rdc, float tol, int max_iter, float lo, float hi,
                                       float* delta_out, float* rdc_out, int* iters_out, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  if (!d_tokens || !delta_out || !rdc_out || !iters_out) return fail(m, ADEPT_ERR_INVALID_ARG, "NULL pointer");
  if (!(target_rdc >= 0.f && target_rdc < 1.f) || !(tol >= 0.f) || max_iter < 1 || !(lo < hi))
    return fail(m, ADEPT_ERR_INVALID_ARG, "calibration needs target in [0, 1), tol >= 0, max_iter >= 1, lo < hi");
  if (batch < 1 || prompt_len < 1) return fail(m, ADEPT_ERR_INVALID_ARG, "batch and prompt_len must be positive");
  const long long T = (long long)batch * prompt_len;
  if (T > m->T_max) return fail(m, ADEPT_ERR_CAPACITY, "calibration batch above the pass workspace");
  cudaStream_t st = (cudaStream_t)stream;
  if (!m->calib_exit) TRY(dalloc_t(m, &m->calib_exit, (size_t)m->T_max));
  std::vector<int32_t> ex((size_t)T);
  float delta = lo;
  double rdc = 0.0;
  int it = 0;
  while (it < max_iter) {
    delta = 0.5f * (lo + hi);
    TRY(adept_prefill(m, batch, prompt_len, d_tokens, delta, nullptr, m->calib_exit, nullptr, nullptr, nullptr, stream));
    CUDA_TRY(m, cudaMemcpyAsync(ex.data(), m->calib_exit, (size_t)T * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
    TRY(adept_check_device_status(m, stream));   // synchronises the stream
    ++it;
    long long depth = 0;
    for (long long j = 0; j < T; ++j) depth += ex[(size_t)j];
    rdc = 1.0 - (double)depth / ((double)T * m->N);
    if (std::fabs(rdc - (double)target_rdc) <= (double)tol) break;
    if (rdc > (double)target_rdc)
      lo = delta;
    else
      hi = delta;
  }
  *delta_out = delta;
  *rdc_out = (float)rdc;
  *iters_out = it;
  return ADEPT_OK;
}

adept_status adept_skip_kv_fill(adept_model* m, int n_tokens, const void* d_h_mapped, const int32_t* d_exit_layer,
                                const int32_t* d_seq, const int32_t* d_pos, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (n_tokens < 0) return fail(m, ADEPT_ERR_INVALID_ARG, "n_tokens < 0");
  if (n_tokens == 0) return ADEPT_OK;
  if (n_tokens > (1 << 20)) return fail(m, ADEPT_ERR_CAPACITY, "n_tokens %d above 1<<20", n_tokens);
  if (!d_h_mapped || !d_exit_layer || !d_seq || !d_pos) return fail(m, ADEPT_ERR_INVALID_ARG, "NULL device pointer");
  cudaStream_t st = (cudaStream_t)stream;
  if (n_tokens > m->fill_cap) {
    // grow the fill workspace (outside any timed or captured region by contract)
    for (void* p : {(void*)m->fill_x, (void*)m->fill_tok}) {
      if (!p) continue;
      cudaFree(p);
      m->allocs.erase(std::remove(m->allocs.begin(), m->allocs.end(), p), m->allocs.end());
    }
    m->fill_x = nullptr;
    m->fill_tok = nullptr;
    m->fill_cap = 0;   // until both buffers of the new capacity exist
    int cap = std::max(n_tokens, 1024);
    TRY(dalloc(m, &m->fill_x, (size_t)cap * m->D * m->esz));
    TRY(dalloc_t(m, &m->fill_tok, cap));
    if (!m->fill_hist) {
      TRY(dalloc_t(m, &m->fill_hist, m->N + 2));
      TRY(dalloc_t(m, &m->fill_start, m->N + 2));
      TRY(dalloc_t(m, &m->fill_cursor, m->N + 2));
    }
    m->fill_cap = cap;
  }
  m->launches += launch_fill_sort(st, m->dt, d_h_mapped, n_tokens, m->D, d_exit_layer, m->N, m->fill_hist,
                                  m->fill_start, m->fill_cursor, m->fill_tok, m->fill_x, attn_norm_mode(m),
                                  m->cfg.norm_eps, m->err_word);
  std::vector<GemmProblem> probs;
  std::vector<int> mrs;
  for (int r = 2; r <= m->N; ++r) {
    probs.push_back(kv_problem(m, r - 1, m->fill_x, m->fill_cap, DevRange{nullptr, m->fill_start + r, 0}, m->fill_tok, d_seq, d_pos));
    mrs.push_back(n_tokens);
  }
  // algorithmic work of this launch is only known on the device; the benchmark supplies it.
  // A few tokens: one weight-streaming launch over the layers; else the grouped tcgen05 GEMM.
  bool done = false;
  if (m->dt == ADEPT_DTYPE_BF16 && m->use_dg && !m->force_simt && n_tokens <= DG_MAX_M) {
    cudaEvent_t b = nullptr;
    prof_begin(m, ADEPT_PROF_KV_FILL, st, &b);
    done = streaming_gemm_grouped(m, st, probs.data(), (int)probs.size(), n_tokens) >= 0;
    prof_end(m, ADEPT_PROF_KV_FILL, st, b, 0, 0);
    if (done) m->launches += 1;
  }
  if (!done) gemm(m, st, probs.data(), (int)probs.size(), mrs.data(), ADEPT_PROF_KV_FILL);
  span_collect(m, st);
  return check_launch(m);
}

adept_status adept_seq_reserve(adept_model* m, int batch, const int32_t* h_lens) {
  if (!m || !h_lens) return ADEPT_ERR_INVALID_ARG;
  if (batch < 1 || batch > m->cfg.max_batch) return fail(m, ADEPT_ERR_CAPACITY, "batch %d out of range", batch);
  for (int b = 0; b < batch; ++b)
    if (h_lens[b] < 0 || h_lens[b] > m->cfg.max_seq) return fail(m, ADEPT_ERR_INVALID_ARG, "length out of range");
  TRY(reserve_seqs(m, batch, h_lens, 0));
  CUDA_TRY(m, cudaStreamSynchronize(0));
  return ADEPT_OK;
}

adept_status adept_read_kv(adept_model* m, int layer, int seq, int pos0, int n_pos, void* d_k_out, void* d_v_out,
                           void* stream) {
  if (!m || !d_k_out || !d_v_out) return ADEPT_ERR_INVALID_ARG;
  if (layer < 1 || layer > m->N) return fail(m, ADEPT_ERR_INVALID_ARG, "layer %d out of [1, N]", layer);
  if (seq < 0 || seq >= m->cfg.max_batch || m->seq_blocks[seq].empty())
    return fail(m, ADEPT_ERR_INVALID_ARG, "sequence %d not reserved", seq);
  if (pos0 < 0 || n_pos < 0 || pos0 + n_pos > m->max_blocks_per_seq * m->cfg.kv_block_tokens)
    return fail(m, ADEPT_ERR_INVALID_ARG, "position range out of the reserved blocks");
  launch_read_kv((cudaStream_t)stream, m->dt, cache_view(m), layer - 1, seq, pos0, n_pos, d_k_out, d_v_out);
  return check_launch(m);
}

adept_status adept_read_final_states(adept_model* m, float* d_out, int rows, void* stream) {
  if (!m || !d_out) return ADEPT_ERR_INVALID_ARG;
  if (rows < 0 || rows > m->last_rows) return fail(m, ADEPT_ERR_INVALID_ARG, "rows %d > last pass rows", rows);
  CUDA_TRY(m, cudaMemcpyAsync(d_out, m->final_, (size_t)rows * m->D * sizeof(float), cudaMemcpyDeviceToDevice,
                              (cudaStream_t)stream));
  return ADEPT_OK;
}

adept_status adept_check_device_status(adept_model* m, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  CUDA_TRY(m, cudaStreamSynchronize(st));
  CUDA_TRY(m, cudaGetLastError());
  unsigned w = 0;
  CUDA_TRY(m, cudaMemcpy(&w, m->err_word, sizeof w, cudaMemcpyDeviceToHost));
  CUDA_TRY(m, cudaMemset(m->err_word, 0, sizeof(unsigned)));
  if (w & ERRW_TIMEOUT) {
    // a launch that gave up may have left arrival counters of the stream-K GEMM counted
    if (m->ds_cnt) CUDA_TRY(m, cudaMemset(m->ds_cnt, 0, sizeof(int) * DS_CNT_CAP));
    return fail(m, ADEPT_ERR_TIMEOUT, "a device-side wait timed out (word 0x%x)", w);
  }
  if (w) return fail(m, ADEPT_ERR_DEVICE_INPUT, "device-side input check failed (word 0x%x)", w);
  return ADEPT_OK;
}

adept_status adept_set_wait_limit(int64_t cycles) {
  if (cycles < 0) return fail(nullptr, ADEPT_ERR_INVALID_ARG, "wait limit %lld < 0", (long long)cycles);
  const long long v = cycles == 0 ? WAIT_LIMIT_DEFAULT : (long long)cycles;
  for (cudaError_t e : {set_wait_limit_tc(v), set_wait_limit_dg(v), set_wait_limit_ds(v)})
    if (e != cudaSuccess) return fail(nullptr, ADEPT_ERR_CUDA, "setting the wait limit: %s", cudaGetErrorString(e));
  return ADEPT_OK;
}

void adept_set_alloc_fail_after(int64_t n) { g_alloc_budget.store(n < 0 ? -1 : (long long)n); }

adept_status adept_set_option(adept_model* m, int option, int value) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  switch (option) {
    case ADEPT_OPT_HSM_IDENTITY: m->hsm_identity = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_PROFILE: m->profile = value != 0; return ADEPT_OK;
    case ADEPT_OPT_SPAN_TIMER:
      if (value && !m->span_sites) {
        TRY(dalloc_t(m, &m->span_sites, SPAN_SITES));
        TRY(dalloc_t(m, &m->span_tot, ADEPT_PROF_NCLASS));
        const std::vector<SpanSite> idle(SPAN_SITES, SpanSite{~0ull, 0ull, 0, 0});
        CUDA_TRY(m, cudaMemcpy(m->span_sites, idle.data(), SPAN_SITES * sizeof(SpanSite), cudaMemcpyHostToDevice));
        CUDA_TRY(m, cudaMemset(m->span_tot, 0, ADEPT_PROF_NCLASS * sizeof(SpanTotal)));
      }
      m->span_on = value != 0;
      drop_graphs(m);   // captured steps carry their launches' span sites
      return ADEPT_OK;
    case ADEPT_OPT_GEMM_SIMT: m->force_simt = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_DECODE_GRAPH: m->use_graph = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_DECODE_GEMM: m->use_dg = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_DECODE_STREAM: m->use_stream = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_DECODE_TILED: m->use_tiled = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_ATTN_TC: m->use_attn_tc = value != 0; return ADEPT_OK;
    case ADEPT_OPT_FUSED_EXIT: m->use_fused_exit = value != 0; drop_graphs(m); return ADEPT_OK;
    case ADEPT_OPT_EXIT_METRIC:
      if (value < EXIT_GLOBAL || value > EXIT_BOTH) return fail(m, ADEPT_ERR_INVALID_ARG, "exit metric %d", value);
      m->exit_metric = value;
      drop_graphs(m);
      return ADEPT_OK;
    case ADEPT_OPT_ALL_AT_ONCE: m->all_at_once = value != 0; return ADEPT_OK;
    case ADEPT_OPT_STOP_ENTIRELY:
      if (value && (m->cfg.family != ADEPT_FAMILY_BERT || m->dt != ADEPT_DTYPE_BF16))
        return fail(m, ADEPT_ERR_INVALID_ARG, "stop-entirely is defined for bf16 encoder models");
      if (value && !m->tok_exit) TRY(dalloc_t(m, &m->tok_exit, (size_t)m->T_max));
      m->stop_entirely = value != 0;
      return ADEPT_OK;
  }
  return fail(m, ADEPT_ERR_INVALID_ARG, "unknown option %d", option);
}

adept_status adept_span_read(adept_model* m, int cls, int64_t* launches, double* total_ms) {
  if (!m || cls < 0 || cls >= ADEPT_PROF_NCLASS) return ADEPT_ERR_INVALID_ARG;
  if (launches) *launches = 0;
  if (total_ms) *total_ms = 0;
  if (!m->span_tot) return ADEPT_OK;
  CUDA_TRY(m, cudaDeviceSynchronize());
  SpanTotal t{};
  CUDA_TRY(m, cudaMemcpy(&t, m->span_tot + cls, sizeof t, cudaMemcpyDeviceToHost));
  CUDA_TRY(m, cudaMemset(m->span_tot + cls, 0, sizeof t));
  if (launches) *launches = (int64_t)t.n;
  if (total_ms) *total_ms = (double)t.ns * 1e-6;
  return ADEPT_OK;
}

adept_status adept_profile_read(adept_model* m, int cls, int64_t* launches, double* total_ms, double* flops,
                                double* bytes) {
  if (!m || cls < 0 || cls >= ADEPT_PROF_NCLASS) return ADEPT_ERR_INVALID_ARG;
  CUDA_TRY(m, cudaDeviceSynchronize());
  ProfRec& pr = m->prof[cls];
  double ms = 0, fl = 0, by = 0;
  for (size_t i = 0; i < pr.ev.size(); ++i) {
    float t = 0;
    cudaEventElapsedTime(&t, pr.ev[i].first, pr.ev[i].second);
    ms += t;
    fl += pr.work[i].first;
    by += pr.work[i].second;
  }
  if (launches) *launches = (int64_t)pr.ev.size();
  if (total_ms) *total_ms = ms;
  if (flops) *flops = fl;
  if (bytes) *bytes = by;
  pr.ev.clear();
  pr.work.clear();
  bool any = false;
  for (auto& q : m->prof) any |= !q.ev.empty();
  if (!any) m->ev_used = 0;   // every recorded pair was read: the pool can be reused
  return ADEPT_OK;
}

adept_status adept_hsm_train_init(adept_model* m, int max_rows, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (max_rows < 1) return fail(m, ADEPT_ERR_INVALID_ARG, "max_rows %d < 1", max_rows);
  if (m->cfg.family == ADEPT_FAMILY_BERT && (m->cfg.n_classes < 1 || m->cfg.n_classes > HT_MAX_CLASSES))
    return fail(m, ADEPT_ERR_INVALID_ARG, "encoder HSM training needs n_classes in [1, %d]", HT_MAX_CLASSES);
  if (m->dt == ADEPT_DTYPE_BF16 && ((m->D | m->m1 | m->m2) & 7))
    return fail(m, ADEPT_ERR_INVALID_ARG, "bf16 HSM training needs D, m1, m2 multiples of 8");
  const adept_status s = ht_init(m, max_rows, (cudaStream_t)stream);
  if (s != ADEPT_OK) ht_free(m);
  return s;
}

adept_status adept_hsm_train_step(adept_model* m, int n, const float* d_s_i, const float* d_s_prev,
                                  const float* d_inertia, const int32_t* d_target, const adept_adamw* hp,
                                  float* d_loss_out, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (!m->ht) return fail(m, ADEPT_ERR_INVALID_ARG, "adept_hsm_train_init has not run");
  if (m->cfg.family == ADEPT_FAMILY_BERT)
    return fail(m, ADEPT_ERR_INVALID_ARG, "encoders train with adept_hsm_train_step_cls");
  if (n < 1 || n > m->ht->cap) return fail(m, ADEPT_ERR_INVALID_ARG, "n %d outside [1, %d]", n, m->ht->cap);
  if (!d_s_i || !d_s_prev || !d_inertia || !d_target || !hp) return fail(m, ADEPT_ERR_INVALID_ARG, "NULL pointer");
  if (!adamw_ok(hp)) return fail(m, ADEPT_ERR_INVALID_ARG, "AdamW hyperparameters out of range");
  return ht_step(m, n, d_s_i, d_s_prev, d_inertia, d_target, *hp, d_loss_out, (cudaStream_t)stream);
}

adept_status adept_hsm_train_step_cls(adept_model* m, int n, const float* d_s_i, const float* d_s_prev,
                                      const float* d_inertia, const float* d_s_final, int n_cls,
                                      const int32_t* d_label, float cls_weight, const adept_adamw* hp,
                                      float* d_loss_out, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  g_pdl = !m->profile;
  if (!m->ht) return fail(m, ADEPT_ERR_INVALID_ARG, "adept_hsm_train_init has not run");
  if (m->cfg.family != ADEPT_FAMILY_BERT)
    return fail(m, ADEPT_ERR_INVALID_ARG, "decoders train with adept_hsm_train_step");
  if (n < 1 || n > m->ht->cap) return fail(m, ADEPT_ERR_INVALID_ARG, "n %d outside [1, %d]", n, m->ht->cap);
  if (n_cls < 0 || n_cls > n) return fail(m, ADEPT_ERR_INVALID_ARG, "n_cls %d outside [0, %d]", n_cls, n);
  if (!d_s_i || !d_s_prev || !d_inertia || !d_s_final || (n_cls > 0 && !d_label) || !hp)
    return fail(m, ADEPT_ERR_INVALID_ARG, "NULL pointer");
  if (!(cls_weight >= 0.f && cls_weight < INFINITY)) return fail(m, ADEPT_ERR_INVALID_ARG, "cls_weight out of range");
  if (!adamw_ok(hp)) return fail(m, ADEPT_ERR_INVALID_ARG, "AdamW hyperparameters out of range");
  return ht_step_cls(m, n, d_s_i, d_s_prev, d_inertia, d_s_final, n_cls, d_label, cls_weight, *hp, d_loss_out,
                     (cudaStream_t)stream);
}

adept_status adept_hsm_train_read(adept_model* m, int what, int param, float* d_out, int64_t count, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  if (!m->ht) return fail(m, ADEPT_ERR_INVALID_ARG, "adept_hsm_train_init has not run");
  if (param < 0 || param >= HT_NPARAM) return fail(m, ADEPT_ERR_INVALID_ARG, "param %d outside [0, 12]", param);
  const HsmTrain& t = *m->ht;
  const float* base = what == ADEPT_HSM_PARAMS ? t.theta : what == ADEPT_HSM_GRADS ? t.grad
                      : what == ADEPT_HSM_MOMENT1 ? t.mom1 : what == ADEPT_HSM_MOMENT2 ? t.mom2 : nullptr;
  if (!base) return fail(m, ADEPT_ERR_INVALID_ARG, "what %d unknown", what);
  if (!d_out || count != t.numel[param])
    return fail(m, ADEPT_ERR_INVALID_ARG, "count %lld != %lld", (long long)count, t.numel[param]);
  CUDA_TRY(m, cudaMemcpyAsync(d_out, base + t.off[param], (size_t)count * 4, cudaMemcpyDeviceToDevice,
                              (cudaStream_t)stream));
  return ADEPT_OK;
}

int64_t adept_hsm_param_numel(const adept_model* m, int param) {
  if (!m || param < 0 || param >= HT_NPARAM) return -1;
  const int D = m->D, m1 = m->m1, m2 = m->m2;
  const int64_t n[HT_NPARAM] = {D, 9, 1, (int64_t)m1 * D, m1, (int64_t)m2 * m1, m2, (int64_t)m1 * m2, m1, m1,
                                (int64_t)D * m1, D, D};
  return n[param];
}

int64_t adept_launch_count(adept_model* m) {
  if (!m) return 0;
  const int64_t n = m->launches;
  m->launches = 0;
  return n;
}

}  // extern "C"

#ifdef ADEPT_KTRACE
namespace adept {
void kt_attach_attention(void*, unsigned*, unsigned);
void kt_attach_simt(void*, unsigned*, unsigned);
void kt_attach_misc(void*, unsigned*, unsigned);
void kt_attach_tc(void*, unsigned*, unsigned);
void kt_attach_dg(void*, unsigned*, unsigned);
void kt_attach_hsm_train(void*, unsigned*, unsigned);
}  // namespace adept
// Debug build only: points every kernel's timeline records at dev_buf (cap records of 104
// bytes) and the device counter dev_cnt (NULL buffer: recording off).
extern "C" ADEPT_API void adept_debug_ktrace(void* dev_buf, unsigned* dev_cnt, unsigned cap) {
  kt_attach_attention(dev_buf, dev_cnt, cap);
  kt_attach_simt(dev_buf, dev_cnt, cap);
  kt_attach_misc(dev_buf, dev_cnt, cap);
  kt_attach_tc(dev_buf, dev_cnt, cap);
  kt_attach_dg(dev_buf, dev_cnt, cap);
  kt_attach_hsm_train(dev_buf, dev_cnt, cap);
}
#endif


// ---------------------------------------------------------------------------
// Read-only view of a loaded model for the allocation-free fill entry point
// (fill_noalloc.cu).  Copies pointers and sizes only.
// ---------------------------------------------------------------------------
namespace adept {
bool model_fill_view(adept_model* m, FillView* v) {
  if (!m || m->N > FILL_VIEW_MAX_LAYERS) return false;
  v->n_layers = m->N;
  v->d_model = m->D;
  v->d_q = m->Dq;
  v->d_kv = m->Dkv;
  v->head_dim = m->dh;
  v->dtype = m->dt;
  v->norm_mode = attn_norm_mode(m);
  v->norm_eps = m->cfg.norm_eps;
  v->rope = m->cfg.family == ADEPT_FAMILY_LLAMA;
  v->rope_table = m->rope_table;
  v->cache = cache_view(m);
  v->err_word = m->err_word;
  for (int l = 0; l < m->N; ++l) {
    v->w_kv[l] = (const char*)m->L[l].w_qkv + (size_t)m->Dq * m->D * m->esz;
    v->b_kv[l] = m->L[l].b_qkv + m->Dq;
  }
  return true;
}

void model_set_error(adept_model* m, const char* msg) {
  if (m) m->err = msg;
}

void model_add_launches(adept_model* m, int n) {
  if (m) m->launches += n;
}
}  // namespace adept

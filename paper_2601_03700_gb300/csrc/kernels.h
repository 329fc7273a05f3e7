// Host-side launchers of the library's kernels (all enqueue on the given stream).
#pragma once
#include "common.cuh"

namespace adept {

// Device counter word layout of one pass.
// Exit-test similarity (Sec. 4.1 global; App. H.3 local and both).
enum : int { EXIT_GLOBAL = 0, EXIT_LOCAL = 1, EXIT_BOTH = 2 };

enum : int {
  CTR_ACTIVE = 0,    // [0], [1]: active rows, ping-pong by layer parity
  CTR_EXITED = 2,    // exits so far in this pass
  CTR_PREFIX = 3,    // [3 + i]: exits after layer i (i = 0..N)
};
__host__ __device__ static inline int ctr_words(int n_layers) { return CTR_PREFIX + n_layers + 2; }

// The similarity the exit test compares with delta: global cos(s_i, I) (Eq. 7), local
// cos(s_i, s_{i-1}) or both (their minimum: both must reach delta), App. H.3; from the sums
// ns = |s_i|^2, ni = |I|^2, dot = <s_i, I>, np = |s_{i-1}|^2, dp = <s_i, s_{i-1}>.  A zero
// norm gives -inf (never exits).
static __device__ __forceinline__ float exit_similarity(int metric, float ns, float ni, float dot, float np_,
                                                       float dp) {
  const float g = (ns > 0.f && ni > 0.f) ? dot / sqrtf(ns * ni) : -INFINITY;
  if (metric == EXIT_GLOBAL) return g;
  const float l = (ns > 0.f && np_ > 0.f) ? dp / sqrtf(ns * np_) : -INFINITY;
  return metric == EXIT_LOCAL ? l : fminf(g, l);
}

// Token -> (sequence, position) maps, identity row map, the pass's counters (all rows
// active), if sim is given NaN for every (token, layer) similarity, and if tok_exit is
// given N as every token's exit layer so far.
void launch_pass_init(cudaStream_t st, int n_tok, int prompt_len, int decode, int* tok_seq, int* tok_pos,
                      int* row_tok, int* seq_len, int seq_cap, int max_pos, unsigned* err, int* ctr, int n_ctr,
                      float* sim, int n_layers, int* tok_exit);
// xhat (optional, decoders): the embedded rows standardised (smode, seps) in bf16, [n_tok][D].
void launch_embed(cudaStream_t st, int dt, const int* tokens, int n_tok, const int* tok_pos, const void* E,
                  const void* P, const float* type_emb, const float* g, const float* b, int family, int D, int V,
                  float eps, float* X, unsigned* err, bf16* xhat, int smode, float seps);
void launch_standardize(cudaStream_t st, int dt, const float* X, int ldx, const int* in_rows, DevRange rows,
                        int max_rows, int D, int mode, float eps, void* out, int ld_out);
void launch_layernorm_inplace(cudaStream_t st, float* X, DevRange rows, int max_rows, int D, const float* g,
                              const float* b, float eps);
// Exit decisions of the active rows.  metric: EXIT_*; Xin = the layer's input rows s_{i-1}
// (local metric).  The exit kernels below take the same metric and aao_len: all-at-once
// prompt exits (App. H.2) with aao_len = the prompt length (every row takes the decision of
// its sequence's last prompt token; tok_pos gives a token's position), 0 = token level.
void launch_exit_decide(cudaStream_t st, const float* Xout, const float* I, const float* Xin, int D, DevRange rows,
                        int max_rows, const int* row_tok, const int* forced, int layer, int n_layers,
                        const float* delta_p, int test, int metric, float* sim, int* flag, float* inv_norm,
                        unsigned* err);
// Test + compaction + moves in one CTA for passes of at most EXIT_SMALL_MAX rows
// (max_rows: the pass's row bound; at most 16 rows take a register-resident kernel, which
// also writes xhat_next (if given): each kept row standardised (smode, seps) for the next
// layer's attention input, bf16 [new row][D]).  Returns whether the register-resident
// kernel ran (xhat_next written).
constexpr int EXIT_SMALL_MAX = 256;
bool launch_exit_small(cudaStream_t st, const float* Xin, const float* Xout, const float* I, int first, int D,
                       int* ctr, int par, const int* row_tok, int* row_tok_next, const int* forced, int layer,
                       int n_layers, const float* delta_p, int test, float* sim, int* exit_tok, int* exit_layer_out,
                       float* Xnext, float* Inext, float* hsm_s, float* hsm_prev, float* hsm_I, int max_rows,
                       bf16* xhat_next, int smode, float seps, int metric, int aao_len, const int* tok_pos,
                       unsigned* err);
void launch_set_float(cudaStream_t st, float* p, float v);
void launch_span_collect(cudaStream_t st, SpanSite* sites, int n, SpanTotal* tot, int n_cls);
// Generation-step staging of the caller's inputs (forced NULL -> zeros) and outputs (each
// output optional).
void launch_stage_in(cudaStream_t st, float* d_delta, float delta, const int* tokens, int* dec_tok, const int* forced,
                     int* dec_forced, int batch);
void launch_stage_out(cudaStream_t st, int batch, const int* dec_exit, int* exit_out, const int* dec_next,
                      int* next_out, const float* logits, float* logits_out, long long n_logits, const float* sim,
                      float* sim_out, int n_sim);
void launch_exit_scan(cudaStream_t st, int* ctr, int in_parity, const int* flag, const int* row_tok,
                      int* row_tok_next, int* exit_tok, int* dst, int* exit_layer_out, int layer, int aao_len,
                      const int* tok_pos);
void launch_exit_move(cudaStream_t st, const float* Xin, const float* Xout, const float* I, int first, int D,
                      const int* n_rows, int max_rows, const int* dst, const float* inv_norm, float* Xnext,
                      float* Inext, float* hsm_s, float* hsm_prev, float* hsm_I);
void launch_final_scatter(cudaStream_t st, const float* X, int D, const int* n_rows, int max_rows, const int* row_tok,
                          float* final_, int* exit_layer_out, int n_layers);
// launch_final_scatter that also writes each row standardised for the output head (hmode, heps)
// in bf16 at xhead[token] (generation steps); rows of up to 8192 elements (head_rows_supported).
bool head_rows_supported(int D);
void launch_final_scatter_head(cudaStream_t st, const float* X, int D, const int* n_rows, int max_rows,
                               const int* row_tok, float* final_, int* exit_layer_out, int n_layers, bf16* xhead,
                               int hmode, float heps);
void launch_hsm_prep(cudaStream_t st, int dt, const float* hs, const float* hp, const float* hI, DevRange rows,
                     int max_rows, int D, const float* g0, const float* conv, float eps, float* c0f, void* c0t);
void launch_hsm_mid(cudaStream_t st, int dt, const float* h3, const float* h1, DevRange rows, int max_rows, int m1,
                    const float* g1, float eps, void* h4);
// xhead (optional): each row's standardised s~ also at xhead[token] (generation steps' head input).
void launch_hsm_out(cudaStream_t st, int dt, const float* h5, const float* c0f, const float* hs, int identity,
                    DevRange rows, int max_rows, int D, const float* g2, float eps, const int* exit_tok,
                    float* final_, void* xfill, int fill_mode, float norm_eps, void* xhead = nullptr);
// Greedy token per row (lowest index on ties); part_v / part_i: rows * 32 partials.
int launch_argmax(cudaStream_t st, const float* logits, int V, int rows, int* out, float* part_v, int* part_i);
void launch_head_rows(cudaStream_t st, int batch, int prompt_len, int last, int* rows);
// Returns the number of launches (1 for calls of at most 32 tokens, else 2).
int launch_fill_sort(cudaStream_t st, int dt, const void* h, int n, int D, const int* exit_layer, int n_layers,
                     int* hist, int* start, int* cursor, int* sorted_tok, void* xs, int mode, float eps,
                     unsigned* err);
void launch_fold_rows(cudaStream_t st, int dt, void* dst, int ld_dst, const void* src, int n_rows, int K,
                      const float* gamma, const float* beta, const float* bias_in, float* bias_out, int row_mode);
void launch_to_f32(cudaStream_t st, int dt, const void* src, float* dst, int n);
// Writes the tile-contiguous copy (GemmProblem::Bt layout, tiled_bytes(N, K) bytes) of the
// row-major bf16 matrix src [N][K] (row stride ld elements) into dst.
void launch_tile_weight(cudaStream_t st, const void* src, int N, int K, int ld, void* dst);
void launch_read_kv(cudaStream_t st, int dt, KVCacheView c, int layer0, int seq, int pos0, int n_pos, void* ko,
                    void* vo);

// GEMMs.  SIMT path: C = A B^T into fp32 scratch, then the epilogue kernel.
void launch_gemm_simt(cudaStream_t st, int dt, const GemmProblem& p, int max_rows, float* scratch);
// Attention of the active query rows over the paged cache of one layer.
// decode_keys > 0 (generation step, one query row per sequence): split-KV kernel over at
// most decode_keys keys, using ws (>= rows * heads * ATTN_MAX_SPLIT * (head_dim + 2) floats)
// and, for bf16, counters (>= rows * heads ints, zero between launches; the kernel leaves
// them zero).  key_exit (prompt passes, bf16; the encoder's "stop entirely" variant): the
// exit layer so far of each token of the pass (token = sequence * kp_len + position); a key
// whose token left before this layer is left out.
constexpr int ATTN_MAX_SPLIT = 32;
void launch_attention(cudaStream_t st, int dt, const void* q, int ld_q, void* out, int ld_out, DevRange rows,
                      int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos, const int* seq_len,
                      KVCacheView cache, int layer0, int n_heads, int causal, int decode_keys, float* ws,
                      int* counters, unsigned* err, const int* key_exit = nullptr, int kp_len = 0,
                      int q_rows = 0, int n_layers = 0);

}  // namespace adept

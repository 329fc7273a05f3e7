// Persistent generation-step kernel (decode_fused.cu): the whole early-exit step of a
// small batch in one cooperative launch.  Internal interface used by the runtime.
#pragma once
#include "common.cuh"

#include <string>

namespace adept {

constexpr int DF_MAX_BATCH = 16;    // token rows a fused step can carry
constexpr int DF_MAX_LAYERS = 64;   // the fill-group mask is one 64-bit word

struct DfLayerSrc {
  const void* w_qkv;   // [D_q + 2 D_kv, D], gain folded, RoPE pairs adjacent
  const float* b_qkv;
  const void* w_o;     // [D, D_q]
  const float* b_o;
  const void* w_up;    // [up_rows, D] (SwiGLU: gate / up interleaved by 16 rows)
  const float* b_up;
  int up_rows;
  const void* w_down;  // [D, F]
  const float* b_down;
};

// Everything the fused step reads or writes, as laid out by the runtime.
struct DfModelSrc {
  int N, D, H, Hkv, dh, Dq, Dkv, F, V, m1, m2, family, norm_mode;
  float eps, hsm_eps;
  int max_batch, seq_cap, max_pos;
  const void* tok_emb;
  const void* pos_emb;          // NULL for rotary families
  const DfLayerSrc* L;          // host array of N
  const void* w_head;
  const float* b_head;
  const void *hsm_w1, *hsm_w2, *hsm_w3, *hsm_w4;
  const float *hsm_b1, *hsm_b2, *hsm_b3, *hsm_b4;
  const float *hsm_g0, *hsm_conv, *hsm_g1, *hsm_g2;
  const float2* rope_table;
  KVCacheView cache;
  float* X_in[2];
  float* X_out;
  float* I[2];
  int* row_tok[2];
  int *tok_seq, *tok_pos, *seq_len, *ctr;
  unsigned* err;
  void *q, *att, *hbuf, *xfill, *h1t, *h2t;
  float *hsm_s, *hsm_prev, *hsm_I, *final_, *c0f, *h1f, *h3f, *h5f, *logits;
  int* exit_tok;
};

struct DfState;

// Builds the device plan (weight tensor maps, epilogues, workspaces).  Returns NULL and
// sets *why when the model does not fit the fused step (dtype, family, sizes).
DfState* df_create(const DfModelSrc& s, std::string* why);
void df_destroy(DfState* d);
// Largest batch a fused step takes for this model (0: none).
int df_max_batch(const DfState* d);
// Enqueues one generation step of B sequences (B <= df_max_batch).  h_pos: host array of
// each sequence's position of the new token (its current length).  Outputs may be NULL
// except next_out.  Returns the launch status.
cudaError_t df_step(DfState* d, cudaStream_t st, int B, const int* tokens, const int* forced, float delta,
                    int hsm_identity, const int* h_pos, int* exit_out, float* sim_out, int* next_out);
// Clears the grid-barrier words after a step that gave up on a wait.
void df_reset(DfState* d, cudaStream_t st);
// Grid size of the persistent launch.
int df_grid(const DfState* d);

}  // namespace adept

// Prompt-pass attention on the tcgen05 tensor cores (attention_tc.cu).
#pragma once
#include "common.cuh"

namespace adept {
// Softmax attention of the active query rows (bf16 Q [rows][ld_q], head h at column h * d_h)
// over the paged cache of layer layer0 (n_layers layers in the pools), causal or over all
// seq_len[seq] keys, into out [rows][ld_out] (bf16).  q_rows: rows of the Q buffer (the TMA
// view's extent).  Returns the launches (1), 0 for no rows, or -1 when the shape is not taken
// (d_h other than 64 / 128, a row range with a device start, no tensor-core device).
int launch_attention_tc(cudaStream_t st, const void* q, int ld_q, int q_rows, void* out, int ld_out, DevRange rows,
                        int max_rows, const int* row_tok, const int* tok_seq, const int* tok_pos, const int* seq_len,
                        const KVCacheView& cache, int n_layers, int layer0, int n_heads, int causal, float scale_log2,
                        unsigned* err);
}  // namespace adept

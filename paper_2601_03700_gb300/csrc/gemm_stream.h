// Stream-K weight-streaming GEMM for passes of at most 16 token rows (gemm_stream.cu).
#pragma once
#include "common.cuh"
#include "gemm_decode.h"

namespace adept {

// Device workspace of the stream-K GEMM, owned by the caller (one per model):
//  part  fp32 partial tiles, [2 * grid][16][32] (two slots per CTA: its first and its last
//        tile, when that tile is shared with another CTA)
//  cnt   arrival counters, one per (problem, tile) of a launch; zero between launches (the
//        last arriving CTA of a tile resets its counter)
struct DsWork {
  float* part;
  int part_ctas;   // CTAs the partial buffer has slots for
  int* cnt;
  int cnt_cap;     // counters available
};

// Bytes of the two buffers for a GPU with `sms` SMs.
size_t stream_gemm_part_bytes(int sms);
constexpr int DS_CNT_CAP = 16384;

// Enqueues one problem (or, grouped, n <= 32 EPI_KV problems of one shape that share A and
// differ in weights, row count and epilogue) on the stream-K kernel.  Returns the number of
// launches (1), or -1 when the shape is not taken (the caller runs another path): more than
// 16 rows, K not a multiple of 64, the A rows do not fit in shared memory, too few weight
// bytes for a stream (the cluster K-split kernel is faster there), or too many tiles.
int stream_gemm(cudaStream_t st, const GemmProblem& p, int max_rows, const DgNorm* norm, const DsWork& ws,
                unsigned* err);

// The previous layer's exit step (Sec. 4.1 exit test, inertia update and stable compaction;
// App. I) taken into the next layer's QKV launch of a generation step, in place of the
// separate exit kernel.  The layer's rows are those of ctr[CTR_ACTIVE + par] / row_tok (at most
// DS_EXIT_MAX_ROWS); every CTA reduces them in the same order and takes the same decisions, CTA
// 0 writes the pass's records (counters, compaction, exit records, similarities), every CTA its
// slice of the moved rows (the kept rows' state and inertia; the leaving rows' mapper inputs), and
// the kept rows, standardised, are the launch's A operand.  The global similarity of Sec. 4.1
// only (the local rules of App. H.3 keep the exit kernel).  The exits before layer i are read
// from ctr[CTR_PREFIX + layer - 1] (written by the previous layer's exit step), so no CTA reads a
// counter another CTA of the launch writes.
constexpr int DS_EXIT_MAX_ROWS = 4;
struct DsExit {
  const float* Xin;    // s_{i-1} of the layer's rows [rows][D]
  const float* Xout;   // s_i
  const float* I;      // inertia before layer i (unused when first)
  float* Xnext;        // kept rows' s_i, compacted
  float* Inext;        // kept rows' inertia after layer i, compacted
  float* hsm_s;        // leaving rows at their exit slot: s_i, s_{i-1}, inertia
  float* hsm_prev;
  float* hsm_I;
  int* ctr;
  const int* row_tok;  // the layer's rows' tokens
  int* row_tok_next;   // the kept rows' tokens, compacted
  const int* forced;   // forced exit layer per token, or NULL
  const float* delta;  // the threshold (device)
  float* sim;          // similarities [token][layer], or NULL
  int* exit_tok;       // exit slot -> token
  int* exit_layer;     // token -> exit layer, or NULL
  unsigned* err;
  int par, layer, n_layers, first, test, metric, norm_mode;
  float eps;
};
// The QKV product (EPI_QKV, one problem) with the exit step of `ex` (p.A is unused: the operand
// is ex->Xout's kept rows, standardised).  -1 when not taken (the caller runs the exit kernel and
// the product separately): the stream-K kernel does not take the shape, more than
// DS_EXIT_MAX_ROWS rows, rows that do not fit in registers, or a local exit rule.
int stream_gemm_exit(cudaStream_t st, const GemmProblem& p, int max_rows, const DsExit& ex, const DsWork& ws,
                     unsigned* err);
int stream_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n, int max_rows, const DsWork& ws,
                        unsigned* err);

}  // namespace adept

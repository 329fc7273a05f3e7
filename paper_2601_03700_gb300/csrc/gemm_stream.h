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
int stream_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n, int max_rows, const DsWork& ws,
                        unsigned* err);

}  // namespace adept

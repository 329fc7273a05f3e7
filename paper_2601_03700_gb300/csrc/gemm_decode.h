// Generation-step GEMM (gemm_decode.cu): C[M, N] = A[M, K] * W[N, K]^T for passes of at
// most DG_MAX_M token rows, shaped as a stream over the weights.
#pragma once
#include "common.cuh"

namespace adept {

constexpr int DG_MAX_M = 16;

// Optional fused standardisation of the A operand: row r of A is the standardised row
// in_rows[r] (or r) of the fp32 matrix X (row length K), as the standardisation kernel
// computes it (LayerNorm without gain / RMS / copy; gains are folded into W at load).
struct DgNorm {
  const float* X;
  int ldx;
  const int* in_rows;
  int mode;     // NormMode
  float eps;
  // Row statistics computed by the producer of X (optional; else computed here from the
  // whole rows): row_stats, (mu, rstd) per row; or tile_stats, [row][K / 32] (mean, M2)
  // of each 32-column tile, merged here in tile order.
  const float2* row_stats;
  const float2* tile_stats;
};

// Enqueues one problem (bf16 operands, fused epilogue).  norm == NULL: A is bf16 at
// p.A.  Returns the number of launches (1), or -1 when the shape is not taken (the caller
// runs another path): max_rows > DG_MAX_M, K not a multiple of 64, K above 16384,
// unaligned operands.
int decode_gemm(cudaStream_t st, const GemmProblem& p, int max_rows, const DgNorm* norm, unsigned* err);
// Whether decode_gemm takes the problem (host-side shape and alignment checks only).
bool decode_gemm_supported(const GemmProblem& p, int max_rows, const DgNorm* norm);
// n (<= 32) cache-fill problems (EPI_KV) of one shape that differ only in their weights, row
// range (rows [0, end)) and epilogue (layer, bias), as one launch (blockIdx.y = problem).
// Returns 1, or -1 when not taken (the caller runs another path).
int decode_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n, int max_rows, unsigned* err);

}  // namespace adept

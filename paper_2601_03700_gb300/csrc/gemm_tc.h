// Grouped tcgen05 GEMM (sm_103a): C[M, N] = A[M, K] * B[N, K]^T per problem, operands
// staged by TMA, fp32 accumulators in tensor memory, fused epilogues (common.cuh).
#pragma once
#include "common.cuh"

namespace adept {
// True when the tensor-core path can run (bf16 operands, sm_100-family device).
bool tc_gemm_supported();
// Enqueues the problems as one grouped launch; returns the number of kernels launched.
int tc_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows, unsigned* err_word);
// As tc_gemm_grouped, without the tensor-map cache (nothing is allocated on any heap).
int tc_gemm_grouped_nocache(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows,
                            unsigned* err_word);
}  // namespace adept

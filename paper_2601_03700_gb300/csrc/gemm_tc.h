// Grouped tcgen05 GEMM (sm_103a): C[M, N] = A[M, K] * B[N, K]^T per problem, operands
// staged by TMA, fp32 accumulators in tensor memory, fused epilogues (common.cuh).
#pragma once
#include "common.cuh"

#include <cuda.h>

namespace adept {
// True when the tensor-core path can run (bf16 operands, sm_100-family device).
bool tc_gemm_supported();
// Enqueues the problems as one grouped launch; returns the number of kernels launched.
int tc_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows, unsigned* err_word);
// As tc_gemm_grouped, without the tensor-map cache (nothing is allocated on any heap).
int tc_gemm_grouped_nocache(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows,
                            unsigned* err_word);
// 2-D view {inner, outer} of a row-major bf16 matrix (row pitch row_bytes) with box
// {64, box_outer}, 128-byte swizzle; cached like the GEMM's own maps.  False if unsupported.
bool tc_encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                  uint32_t box_outer);
// 3-D view {64, rows, K/64} of a K-major bf16 matrix with box {64, box_rows, kc}, 128-byte
// swizzle: one copy brings kc 64-wide k chunks of box_rows rows.  False if unsupported.
bool tc_encode_weight_3d(CUtensorMap* m, const void* base, int K, int rows, size_t row_bytes, int box_rows, int kc);
}  // namespace adept

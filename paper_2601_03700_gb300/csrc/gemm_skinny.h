// Skinny grouped GEMM (at most SKINNY_MAX_M token rows) on bf16 tensor cores.
#pragma once
#include "common.cuh"

namespace adept {
constexpr int SKINNY_MAX_M = 32;
// Enqueues the problems as one launch.  ws: fp32 partial-tile workspace (ws_floats),
// counters: per-tile arrival counters, zero on entry and left zero.  Returns the number
// of kernels launched, or -1 if a problem does not fit this path.
int skinny_gemm_grouped(cudaStream_t st, const GemmProblem* probs, int n_probs, const int* max_rows, float* ws,
                        size_t ws_floats, int* counters, int n_counters);
}  // namespace adept

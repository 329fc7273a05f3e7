// Internal read-only view of a loaded model, for entry points that live outside the
// runtime translation unit.
#pragma once
#include "adept.h"
#include "common.cuh"

namespace adept {
constexpr int FILL_VIEW_MAX_LAYERS = 256;

struct FillView {
  int n_layers, d_model, d_q, d_kv, head_dim, dtype, norm_mode, rope;
  float norm_eps;
  const float2* rope_table;
  KVCacheView cache;
  unsigned* err_word;
  const void* w_kv[FILL_VIEW_MAX_LAYERS];   // layer r-1: the K and V rows of W_qkv (gain folded), [2 D_kv, D]
  const float* b_kv[FILL_VIEW_MAX_LAYERS];  // layer r-1: K and V biases
};

bool model_fill_view(adept_model* m, FillView* v);
void model_set_error(adept_model* m, const char* msg);
// Adds n kernel launches to the model's count (adept_launch_count).
void model_add_launches(adept_model* m, int n);
}  // namespace adept

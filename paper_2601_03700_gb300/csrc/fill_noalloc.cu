// adept_skip_kv_fill_noalloc: the skipped-layer KV fill for callers that cannot
// allocate device memory.
//
// adept_skip_kv_fill keeps its working set (the standardised, exit-layer-sorted copy of
// the mapped states and the bucket counters) in a per-model buffer that it grows with
// cudaMalloc / cudaFree when a call brings more tokens than before.  Some callers cannot
// allow that: code recording a CUDA graph (allocation and the device synchronisation of
// cudaFree are not capturable), serving loops that run under a fixed memory budget or a
// custom allocator, and latency-critical paths where an implicit device synchronisation
// is not acceptable.  This entry point does the same work with its working set in the
// file-scope array below, whose size is fixed when the library is loaded.
//
// The array is shared by every call on a device and keeps the last call's contents; the
// bucket counters that must start at zero are cleared by each call.  Calls that overlap
// on the GPU (different streams, or different models on one device) race on it.
#include "adept.h"
#include "common.cuh"
#include "gemm_tc.h"
#include "kernels.h"
#include "model_view.h"

#include <cstdio>
#include <cstring>
#include <mutex>

namespace adept {

// Working set of one call: standardised mapped states (n x D, model dtype), then the
// sorted token indices (n ints), then three bucket arrays of FILL_VIEW_MAX_LAYERS + 2 ints.
constexpr size_t NOALLOC_SCRATCH_BYTES = ADEPT_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_fill_scratch[NOALLOC_SCRATCH_BYTES];

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Device address of g_fill_scratch per device, looked up once with that device current.
static void* g_scratch_ptr[64];
static std::once_flag g_scratch_once[64];
static cudaError_t g_scratch_err[64];

static void* scratch_address(int dev, cudaError_t* err) {
  if (dev < 0 || dev >= 64) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::call_once(g_scratch_once[dev], [dev] {
    void* p = nullptr;
    g_scratch_err[dev] = cudaGetSymbolAddress(&p, g_fill_scratch);
    g_scratch_ptr[dev] = g_scratch_err[dev] == cudaSuccess ? p : nullptr;
  });
  *err = g_scratch_err[dev];
  return g_scratch_ptr[dev];
}

}  // namespace adept

using namespace adept;

extern "C" ADEPT_API adept_status adept_skip_kv_fill_noalloc(adept_model* m, int n_tokens, const void* d_h_mapped,
                                                             const int32_t* d_exit_layer, const int32_t* d_seq,
                                                             const int32_t* d_pos, void* stream) {
  if (!m) return ADEPT_ERR_INVALID_ARG;
  // launches chain by programmatic dependent launch (this entry point records no profiling
  // events); the calling thread's setting is restored on return
  PdlScope pdl_scope(true);
  if (n_tokens < 0) {
    model_set_error(m, "n_tokens < 0");
    return ADEPT_ERR_INVALID_ARG;
  }
  if (n_tokens == 0) return ADEPT_OK;
  if (!d_h_mapped || !d_exit_layer || !d_seq || !d_pos) {
    model_set_error(m, "NULL device pointer");
    return ADEPT_ERR_INVALID_ARG;
  }
  FillView v;  // on the stack (about 4 KB): nothing on the heap, nothing shared between threads
  if (!model_fill_view(m, &v)) {
    model_set_error(m, "adept_skip_kv_fill_noalloc: model has more layers than the fixed view holds");
    return ADEPT_ERR_INVALID_ARG;
  }
  if (v.dtype != ADEPT_DTYPE_BF16 || !tc_gemm_supported()) {
    model_set_error(m, "adept_skip_kv_fill_noalloc: needs a bf16 model on an sm_100-family GPU");
    return ADEPT_ERR_INVALID_ARG;
  }
  const size_t x_bytes = align256((size_t)n_tokens * v.d_model * 2);
  const size_t tok_bytes = align256((size_t)n_tokens * sizeof(int));
  const size_t bucket_bytes = align256(3 * (size_t)(FILL_VIEW_MAX_LAYERS + 2) * sizeof(int));
  if (x_bytes + tok_bytes + bucket_bytes > NOALLOC_SCRATCH_BYTES) {
    char msg[200];
    snprintf(msg, sizeof msg,
             "adept_skip_kv_fill_noalloc: %d tokens need %zu bytes of scratch, above the fixed %zu bytes "
             "(at most %zu tokens of d_model %d)",
             n_tokens, x_bytes + tok_bytes + bucket_bytes, NOALLOC_SCRATCH_BYTES,
             (NOALLOC_SCRATCH_BYTES - bucket_bytes - 512) / ((size_t)v.d_model * 2 + sizeof(int)), v.d_model);
    model_set_error(m, msg);
    return ADEPT_ERR_CAPACITY;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    model_set_error(m, "adept_skip_kv_fill_noalloc: cudaGetDevice failed");
    return ADEPT_ERR_CUDA;
  }
  cudaError_t se;
  unsigned char* base = (unsigned char*)scratch_address(dev, &se);
  if (!base) {
    model_set_error(m, "adept_skip_kv_fill_noalloc: cudaGetSymbolAddress of the scratch array failed");
    return ADEPT_ERR_CUDA;
  }
  void* xs = base;
  int* sorted_tok = (int*)(base + x_bytes);
  int* hist = (int*)(base + x_bytes + tok_bytes);
  int* start = hist + (FILL_VIEW_MAX_LAYERS + 2);
  int* cursor = start + (FILL_VIEW_MAX_LAYERS + 2);
  cudaStream_t st = (cudaStream_t)stream;
  // bucket by exit layer (the histogram is rebuilt here), standardise s~ once
  model_add_launches(m, launch_fill_sort(st, v.dtype, d_h_mapped, n_tokens, v.d_model, d_exit_layer, v.n_layers, hist,
                                         start, cursor, sorted_tok, xs, v.norm_mode, v.norm_eps, v.err_word));
  // layer r's rows are the sorted prefix with i* < r; groups of at most 32 layers per launch
  GemmProblem probs[32];
  int max_rows[32];
  int np = 0;
  for (int r = 2; r <= v.n_layers; ++r) {
    GemmProblem& p = probs[np];
    memset(&p, 0, sizeof p);
    p.A = xs;
    p.lda = v.d_model;
    p.a_rows = n_tokens;
    p.B = v.w_kv[r - 1];
    p.ldb = v.d_model;
    p.rows = DevRange{nullptr, start + r, 0};
    p.N = 2 * v.d_kv;
    p.K = v.d_model;
    p.epi.kind = EPI_KV;
    p.epi.bias = v.b_kv[r - 1];
    p.epi.row_tok = sorted_tok;
    p.epi.tok_seq = d_seq;
    p.epi.tok_pos = d_pos;
    p.epi.cache = v.cache;
    p.epi.layer0 = r - 1;
    p.epi.n_q_cols = 0;
    p.epi.n_kv_cols = v.d_kv;
    p.epi.head_dim = v.head_dim;
    p.epi.rope = v.rope;
    p.epi.rope_table = v.rope_table;
    max_rows[np] = n_tokens;
    ++np;
    if (np == 32 || r == v.n_layers) {
      const int nl = tc_gemm_grouped_nocache(st, probs, np, max_rows, v.err_word);
      if (nl < 0) {
        model_set_error(m, "adept_skip_kv_fill_noalloc: tensor-core launch rejected the shapes");
        return ADEPT_ERR_INVALID_ARG;
      }
      model_add_launches(m, nl);
      np = 0;
    }
  }
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    model_set_error(m, "adept_skip_kv_fill_noalloc: kernel launch failed");
    return ADEPT_ERR_CUDA;
  }
  return ADEPT_OK;
}

// Shared device-side definitions of the ADEPT GB300 library.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <utility>

typedef __nv_bfloat16 bf16;

// Device error word bits (read by adept_check_device_status).
enum : unsigned {
  ERRW_FORCED = 1u,    // forced exit layer outside {0} U [2, N]
  ERRW_TOKEN = 2u,     // token id outside [0, vocab)
  ERRW_POS = 4u,       // position outside the sequence's reserved blocks / max_pos
  ERRW_EXIT_LAYER = 8u,// exit layer outside [1, N] (skipped-layer fill input)
  ERRW_TIMEOUT = 16u,  // a bounded device-side wait gave up
  ERRW_CONFIG = 32u,   // a kernel was launched with a shape it does not support
  ERRW_LABEL = 64u     // class label outside [0, n_classes)
};

// Programmatic dependent launch.  Every kernel of the library begins with PDL_ENTRY: it
// waits until the kernels it depends on have completed and their writes are visible (a no-op
// when it was launched without the programmatic attribute), then lets the next kernel of the
// stream be launched, so that kernel's launch and prologue overlap this one.  Work placed
// before the wait may touch nothing a preceding kernel writes.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Debug-only launch timeline (built with -DADEPT_KTRACE): thread 0 of every CTA records
// its global-timer stamps at entry, after the dependency wait and at exit, with a kernel
// id (translation unit x 100000 + source line of the entry macro).  Each translation unit
// holds its own pointer to the host-allocated record buffer (set by kt_attach_<unit>).
#ifdef ADEPT_KTRACE
constexpr int KT_MARKS = 8;
struct KtRec {
  unsigned long long t0, t1, t2;
  unsigned long long mk[KT_MARKS];   // optional intermediate stamps (0: not reached)
  unsigned kid, cta, grid, pad;
};
static __device__ KtRec* g_kt_buf = nullptr;
static __device__ unsigned* g_kt_cnt = nullptr;
static __device__ unsigned g_kt_cap = 0;
__device__ __forceinline__ unsigned long long kt_now() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Intermediate marks are SM cycles since the dependency wait (clock64: fine-grained, valid
// within one CTA), stored + 1 so that 0 means "not reached".
__device__ __forceinline__ long long kt_clk() {
  long long c;
  asm volatile("mov.u64 %0, %%clock64;" : "=l"(c));
  return c;
}
struct KtScope {
  unsigned long long t0, t1;
  long long c1;
  unsigned long long mk[KT_MARKS];
  unsigned kid;
  __device__ explicit KtScope(unsigned k) : t0(kt_now()), t1(0), c1(kt_clk()), kid(k) {
#pragma unroll
    for (int i = 0; i < KT_MARKS; ++i) mk[i] = 0;
  }
  __device__ void waited() {
    t1 = kt_now();
    c1 = kt_clk();
  }
  __device__ void mark(int i) { mk[i] = (unsigned long long)(kt_clk() - c1) + 1; }
  __device__ void add(int i, unsigned long long v) { mk[i] += v; }
  __device__ ~KtScope() {
    if (threadIdx.x == 0 && threadIdx.y == 0 && g_kt_buf) {
      const unsigned i = atomicAdd(g_kt_cnt, 1u);
      if (i < g_kt_cap) {
        KtRec r;
        r.t0 = t0;
        r.t1 = t1;
        r.t2 = kt_now();
#pragma unroll
        for (int j = 0; j < KT_MARKS; ++j) r.mk[j] = mk[j];
        r.kid = kid;
        r.cta = blockIdx.x + blockIdx.y * gridDim.x;
        r.grid = gridDim.x * gridDim.y;
        r.pad = 0;
        g_kt_buf[i] = r;
      }
    }
  }
};
#ifndef ADEPT_TU_ID
#define ADEPT_TU_ID 0
#endif
#define KT_BEGIN() KtScope kt_scope_(ADEPT_TU_ID * 100000u + __LINE__)
#define KT_WAITED() kt_scope_.waited()
#define KT_MARK(i) kt_scope_.mark(i)
#define KT_ADD(i, v) kt_scope_.add(i, v)
#define ADEPT_KTRACE_ATTACH(unit)                                                          \
  void kt_attach_##unit(void* buf, unsigned* cnt, unsigned cap) {                          \
    KtRec* b = (KtRec*)buf;                                                                \
    cudaMemcpyToSymbol(g_kt_buf, &b, sizeof b);                                            \
    cudaMemcpyToSymbol(g_kt_cnt, &cnt, sizeof cnt);                                        \
    cudaMemcpyToSymbol(g_kt_cap, &cap, sizeof cap);                                        \
  }
#else
#define KT_BEGIN() \
  do {             \
  } while (0)
#define KT_WAITED() \
  do {              \
  } while (0)
#define KT_MARK(i) \
  do {             \
  } while (0)
#define KT_ADD(i, v) \
  do {               \
  } while (0)
#define ADEPT_KTRACE_ATTACH(unit)
#endif

#define PDL_ENTRY()          \
  KT_BEGIN();                \
  pdl_wait();                \
  KT_WAITED();               \
  pdl_launch_dependents()

// Limit of the library's bounded waits on pipeline progress (a ring slot filling or being
// released, an accumulator becoming ready), in SM cycles; adept_set_wait_limit changes it.
// Each translation unit holds its own copy, set through its set_wait_limit_* function.  The
// waits that let a CTA's copies in flight land before it exits, and the waits of a cluster's
// reduction, keep fixed limits: they must outlast any peer's shortened wait.
constexpr long long WAIT_LIMIT_DEFAULT = 4000000000LL;   // ~2 s at 2 GHz
static __device__ long long g_wait_limit = WAIT_LIMIT_DEFAULT;
// Read once per CTA at kernel entry (a global load; the waits then compare against a register).
__device__ __forceinline__ long long wait_limit() { return g_wait_limit; }
#define ADEPT_WAIT_LIMIT_SETTER(unit)                                               \
  cudaError_t set_wait_limit_##unit(long long cycles) {                              \
    return cudaMemcpyToSymbol(g_wait_limit, &cycles, sizeof cycles);                \
  }

namespace adept {
// In-situ launch spans of the weight-streaming kernels (the span timer option).  A launch's
// span runs from the first of its CTAs past the grid-dependency wait to the end of its last
// CTA.  Every kernel of a stream passes its dependency wait only after its predecessor has
// completed, so the spans of consecutive launches do not overlap and their sum never exceeds
// the elapsed time of the sequence; bytes a kernel fetched before its wait (weights prefetched
// while the predecessor still ran) fall outside its span.  Each CTA's last thread folds its
// stamps into the launch's site with two non-returning reductions (nothing waits on them);
// span_collect_kernel, launched at the end of the pass, adds every used site to its class total
// and resets it.
struct SpanSite {
  unsigned long long t0;   // earliest post-wait stamp of the launch (all ones when idle)
  unsigned long long t1;   // latest CTA end (0 when idle)
  int cls;                 // kernel class of the launch
  int pad;
};
struct SpanTotal {
  unsigned long long ns, n;   // summed spans, launches
};
struct SpanCtx {
  SpanSite* site;    // NULL: not recorded
  int cls;
};
// The span context the weight-streaming launch functions copy into their parameters (set by
// the runtime around a launch on the calling thread; NULL site when the timer is off).
extern thread_local SpanCtx g_span;

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Per-thread recorder: construct at kernel entry, call init() before the CTA's first barrier
// and waited() right after the dependency wait; the destructor (every exit path of every
// thread) counts the thread out, and the CTA's last thread records the CTA's stamps.
struct SpanScope {
  SpanCtx ctx;
  unsigned* left;            // shared: threads of the CTA still running
  unsigned long long* t0s;   // shared: the CTA's post-wait stamp
  __device__ SpanScope(const SpanCtx& c, unsigned* l, unsigned long long* t) : ctx(c), left(l), t0s(t) {}
  __device__ void init() const {
    if (ctx.site && threadIdx.x == 0) *left = blockDim.x * blockDim.y;
  }
  __device__ void waited() const {
    if (ctx.site && threadIdx.x == 0) *t0s = global_ns();
  }
  __device__ ~SpanScope();
};
// Out of line: each exit path carries only the test and the call.
static __device__ __noinline__ void span_close(SpanCtx ctx, unsigned* left, unsigned long long* t0s) {
  __threadfence_block();
  if (atomicSub(left, 1u) != 1u) return;   // not the CTA's last thread
  const unsigned long long t1 = global_ns();
  asm volatile("red.relaxed.gpu.global.min.u64 [%0], %1;" ::"l"(&ctx.site->t0), "l"(*t0s) : "memory");
  asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;" ::"l"(&ctx.site->t1), "l"(t1) : "memory");
  if (blockIdx.x == 0 && blockIdx.y == 0) ctx.site->cls = ctx.cls;
}
__device__ __forceinline__ SpanScope::~SpanScope() {
  if (ctx.site) span_close(ctx, left, t0s);
}

cudaError_t set_wait_limit_tc(long long cycles);
cudaError_t set_wait_limit_dg(long long cycles);
cudaError_t set_wait_limit_ds(long long cycles);

// Launches with the programmatic-serialisation attribute while g_pdl is set (each entry
// point sets it for its calling thread; it is off while per-launch profiling events are
// recorded, so each timed interval holds one kernel alone).
extern thread_local bool g_pdl;
// Sets g_pdl for the calling thread for one scope and restores the previous value on exit.
struct PdlScope {
  bool prev;
  explicit PdlScope(bool on) : prev(g_pdl) { g_pdl = on; }
  ~PdlScope() { g_pdl = prev; }
  PdlScope(const PdlScope&) = delete;
  PdlScope& operator=(const PdlScope&) = delete;
};
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
}  // namespace adept

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f<bf16>(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Block-wide sum for blockDim.x a multiple of 32 (<= 1024); `red` holds 32 floats.
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  float t = (threadIdx.x < (unsigned)nw) ? red[threadIdx.x] : 0.f;
  if (w == 0) t = warp_sum(t);
  if (threadIdx.x == 0) red[0] = t;
  __syncthreads();
  float r = red[0];
  return r;
}

__device__ __forceinline__ float gelu_erf_f(float x) { return 0.5f * x * (1.f + erff(x * 0.70710678118654752f)); }
__device__ __forceinline__ float gelu_tanh_f(float x) {
  return 0.5f * x * (1.f + tanhf(0.79788456080286536f * (x + 0.044715f * x * x * x)));
}
__device__ __forceinline__ float silu_f(float x) { return x / (1.f + expf(-x)); }

enum Act : int { ACT_NONE = 0, ACT_GELU_ERF = 1, ACT_GELU_TANH = 2, ACT_TANH = 3 };
__device__ __forceinline__ float apply_act(int act, float x) {
  switch (act) {
    case ACT_GELU_ERF: return gelu_erf_f(x);
    case ACT_GELU_TANH: return gelu_tanh_f(x);
    case ACT_TANH: return tanhf(x);
    default: return x;
  }
}

// Normalisation applied to a layer's attention input (norm gains / shifts are folded
// into the following projection at load time, so only the standardisation remains).
enum NormMode : int { NORM_RMS = 0, NORM_LN = 1, NORM_COPY = 2 };

// Paged KV cache: pools [n_layers][n_blocks][n_kv_heads][block_tokens][head_dim] for K
// and for V; a sequence's position p lives in block block_table[seq][p / block_tokens].
struct KVCacheView {
  void* k;
  void* v;
  const int* block_table;   // [max_batch][max_blocks_per_seq]
  int max_blocks_per_seq;
  int n_blocks;
  int n_kv_heads;
  int head_dim;
  int block_tokens;
  int max_batch;
  __device__ __forceinline__ size_t offset(int layer0, int seq, int pos, int h) const {
    const int blk = block_table[seq * max_blocks_per_seq + pos / block_tokens];
    return ((((size_t)layer0 * n_blocks + blk) * n_kv_heads + h) * block_tokens + (pos % block_tokens)) *
           (size_t)head_dim;
  }
  // Base offset (head 0, dim 0) of a position, or -1 when (seq, pos) has no reserved block.
  __device__ __forceinline__ long long checked_base(int layer0, int seq, int pos) const {
    if (seq < 0 || seq >= max_batch || pos < 0 || pos >= max_blocks_per_seq * block_tokens) return -1;
    const int blk = block_table[seq * max_blocks_per_seq + pos / block_tokens];
    if (blk < 0 || blk >= n_blocks) return -1;
    return (long long)((((size_t)layer0 * n_blocks + blk) * n_kv_heads) * block_tokens + (pos % block_tokens)) *
           head_dim;
  }
  // Distance between consecutive heads of one position.
  __device__ __forceinline__ size_t head_stride() const { return (size_t)block_tokens * head_dim; }
};

// Row range of a GEMM operand, resolved on the device: rows [*begin, *end) of A (a
// NULL begin means 0; a NULL end means `count`).
struct DevRange {
  const int* begin;
  const int* end;
  int count;
  __device__ __forceinline__ int b() const { return begin ? *begin : 0; }
  __device__ __forceinline__ int e() const { return end ? *end : count; }
};

enum EpiKind : int {
  EPI_F32 = 0,     // out_f32 = acc + bias
  EPI_ACT = 1,     // out_t = act(acc + bias) (and out_f32 if set)
  EPI_RESID = 2,   // out_f32 = resid + acc + bias
  EPI_SWIGLU = 3,  // columns interleaved in 16-blocks (gate, up): out_t = silu(g) * u
  EPI_QKV = 4,     // q -> q_out (RoPE), k/v -> KV cache (RoPE on k)
  EPI_KV = 5       // k/v only (skipped-layer fill) -> KV cache
};

// Epilogue description.  Output row r refers to GEMM row r (relative to the range
// begin); for the cache epilogues its token is row_tok[begin + r].
struct Epi {
  int kind;
  int act;
  const float* bias;
  float* out_f32;
  int ld_f32;
  const float* resid;
  int ld_resid;
  void* out_t;
  int ld_t;
  // QKV / KV
  const int* row_tok;
  const int* tok_seq;
  const int* tok_pos;
  KVCacheView cache;
  int layer0;        // 0-based layer of the cache writes
  int n_q_cols;      // D_q (0 for EPI_KV)
  int n_kv_cols;     // D_kv
  int head_dim;
  int rope;          // apply RoPE to q and k
  const float2* rope_table;   // [max_seq][head_dim/2] (cos, sin)
  // EPI_RESID, generation-step GEMM only (NULL elsewhere): per output row, the (mean, M2)
  // of each 32-column tile of the result, [row][N / 32], for the next standardisation
  float2* tile_stats;
};

// Bits of epi_chunk32's `applied`: work the caller has already done on v.
enum : int { EPI_APPLIED_BIAS_ACT = 1, EPI_APPLIED_RESID = 2 };

// One problem of a (grouped) GEMM: C[M, N] = A[M, K] * B[N, K]^T, both K-major.
struct GemmProblem {
  const void* A;
  int lda;
  int a_rows;       // rows allocated in A (the TMA view's extent; reads past it return zeros)
  const void* B;
  int ldb;
  DevRange rows;
  int N;
  int K;
  Epi epi;
  // rows on the device that are usually far below their bound (the prompt pass's exiting
  // rows): the tensor-core launcher may split the problem by the live count
  int split_live = 0;
  // Optional tile-contiguous copy of B for the weight-streaming kernels (NULL: none): 16 KB
  // units, one per (32-row tile, 256-k block), tile-major, each laid out as the kernels' shared-
  // memory stage (four 64-k chunks of 32 rows x 128 B, 16-byte pieces XOR-swizzled by row & 7,
  // zero past N and K), so that a unit, or a run of its chunks, is one contiguous bulk copy.
  const void* Bt = nullptr;
  int bt_nkb = 0;   // 256-k blocks per tile of Bt
};

static inline int cdiv_h(int a, int b) { return (a + b - 1) / b; }
// Tile-contiguous weight layout (GemmProblem::Bt).
constexpr int TW_ROWS = 32, TW_KB = 256, TW_UNIT = TW_ROWS * TW_KB * 2;
static inline size_t tiled_bytes(int N, int K) { return (size_t)cdiv_h(N, TW_ROWS) * cdiv_h(K, TW_KB) * TW_UNIT; }

static inline int cdiv(int a, int b) { return (a + b - 1) / b; }

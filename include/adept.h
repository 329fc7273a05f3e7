/*
 * adept.h -- C ABI of the GB300 (sm_103a) library for ADEPT's token-level
 * early-exit forward pass (arXiv 2601.03700).
 *
 * Notation follows the paper's problem statement (Sec. 3): N layers, indexed
 * i = 1..N (1-based everywhere in this API), tokens j, hidden size D_h
 * (d_model), query/key/value size D_q (heads x head_dim), exit layer i*.
 *
 * Conventions shared by every call:
 *  - Pointers prefixed d_ are DEVICE pointers owned by the caller; they must stay
 *    valid until the work queued on `stream` has finished.  Pointers prefixed
 *    h_ are host pointers read before the call returns.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Every call that
 *    takes a stream only enqueues work on it and returns; results are valid once
 *    the stream has been synchronised.
 *  - The library owns its copy of the weights, the paged KV cache and its
 *    workspaces (allocated by adept_model_load, released by adept_free).
 *  - Errors are returned as adept_status; nothing is thrown across the ABI.
 *    Argument errors are detected on the host before anything is enqueued.
 *    Device-side input errors (a forced exit layer or token id out of range)
 *    set a device error word that adept_check_device_status reports.
 *    adept_last_error returns a message for the last failing call.
 *  - A model is not thread-safe: calls on one model must be serialised.
 */
#ifndef ADEPT_H
#define ADEPT_H

#include <stdint.h>

#if defined(__GNUC__)
#define ADEPT_API __attribute__((visibility("default")))
#else
#define ADEPT_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ADEPT_OK = 0,
  ADEPT_ERR_INVALID_ARG = 1,   /* bad argument; nothing was enqueued */
  ADEPT_ERR_OOM = 2,           /* device allocation failed */
  ADEPT_ERR_CAPACITY = 3,      /* batch / sequence / KV-block capacity exceeded */
  ADEPT_ERR_CUDA = 4,          /* a CUDA runtime or driver call failed */
  ADEPT_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up */
  ADEPT_ERR_DEVICE_INPUT = 6   /* device-side validation of an input failed */
} adept_status;

enum { ADEPT_FAMILY_LLAMA = 0,   /* RMSNorm pre-norm, RoPE, SwiGLU, untied head */
       ADEPT_FAMILY_GPT2 = 1,    /* LayerNorm pre-norm, learned positions, tanh-GELU, biases, tied head */
       ADEPT_FAMILY_BERT = 2 };  /* post-LN encoder, bidirectional, pooler + classifier */

enum { ADEPT_DTYPE_F32 = 0, ADEPT_DTYPE_BF16 = 1 };

typedef struct {
  int family;          /* ADEPT_FAMILY_* */
  int n_layers;        /* N */
  int d_model;         /* D_h */
  int n_heads;
  int n_kv_heads;      /* 0 -> n_heads */
  int head_dim;        /* D_q = n_heads * head_dim; must be even, <= 128 */
  int d_ffn;
  int vocab;
  int max_pos;         /* learned-position table size (GPT-2 / BERT) */
  int n_classes;       /* encoder classifier outputs */
  int dtype;           /* ADEPT_DTYPE_*: storage and GEMM-input precision; accumulation is fp32 */
  float norm_eps;
  float rope_theta;
  float hsm_eps;       /* eps of the three RMS normalisations inside the HSM */
  int hsm_m1;          /* HSM FC1 / FC3 output width (Table S1: 4 D_h) */
  int hsm_m2;          /* HSM FC2 output width (Table S1: 8 D_h) */
  int kv_block_tokens; /* positions per KV-cache block (16) */
  int max_batch;       /* sequences */
  int max_seq;         /* positions per sequence (prompt + generated) */
  int kv_pool_blocks;  /* 0 -> max_batch * ceil(max_seq / kv_block_tokens) */
  int max_pass_tokens; /* rows of the per-pass workspaces; 0 -> max_batch * max_seq */
  uint64_t block_shuffle_seed; /* 0: KV blocks handed out in order; else a seeded permutation */
  int max_src;         /* > 0 (GPT-2 family only): an encoder-decoder decoder whose layers
                          cross-attend to up to max_src encoder states per sequence
                          (adept_set_cross_source); 0: no cross-attention */
} adept_config;

/* One named weight tensor.  `data` may be a host or a device pointer (it is read
 * with cudaMemcpyDefault); its element type is the model dtype; `numel` must equal
 * the element count of the named shape.  Names (0-based layer slot l = paper layer
 * l+1; matrices are [out, in] row-major):
 *   tok_emb [V,D]; pos_emb [max_pos,D] (GPT-2/BERT); type_emb [D], emb_ln.g/.b [D] (BERT)
 *   layers.l.attn_norm.g/.b, layers.l.ffn_norm.g/.b [D]   (.b not for LLAMA)
 *   layers.l.wq [D_q,D], wk [D_kv,D], wv [D_kv,D], wo [D,D_q]; bq bk bv bo (not LLAMA)
 *   LLAMA: layers.l.w_gate [F,D], w_up [F,D], w_down [D,F]
 *   GPT2/BERT: layers.l.w_fc [F,D], b_fc [F], w_proj [D,F], b_proj [D]
 *   LLAMA: final_norm.g [D], lm_head [V,D]; GPT2: final_norm.g/.b [D] (head tied to tok_emb)
 *   BERT: pool.w [D,D], pool.b [D], cls.w [C,D], cls.b [C]
 *   max_src > 0 (cross-attention sublayer, pre-LN, between self-attention and the FFN):
 *     layers.l.cross_norm.g/.b [D], cwq [D_q,D], cwk [D_kv,D], cwv [D_kv,D], cwo [D,D_q],
 *     cbq cbk cbv cbo
 *   HSM (App. B Table S1): hsm.g0 [D], hsm.conv_w [3,3], hsm.conv_b [1],
 *     hsm.fc1_w [m1,D], hsm.fc1_b, hsm.fc2_w [m2,m1], hsm.fc2_b, hsm.fc3_w [m1,m2],
 *     hsm.fc3_b, hsm.g1 [m1], hsm.fc4_w [D,m1], hsm.fc4_b [D], hsm.g2 [D]      */
typedef struct {
  const char* name;
  const void* data;
  int64_t numel;
} adept_tensor;

typedef struct {
  const adept_tensor* tensors;
  int n_tensors;
} adept_tensor_table;

typedef struct adept_model adept_model;  /* opaque, library-owned */

/* Load a model: validate `cfg`, allocate device memory, copy and repack the weights
 * (norm gains and LN shifts are folded into the following projection), allocate
 * the paged KV pool.  Synchronises `stream` before returning.
 * Errors: INVALID_ARG (bad config, missing or mis-sized tensor), OOM, CUDA. */
ADEPT_API adept_status adept_model_load(const adept_config* cfg, const adept_tensor_table* weights,
                              void* stream, adept_model** out);

/* Prompt pass (prefill) of `batch` sequences of `prompt_len` tokens each; resets
 * sequences 0..batch-1 and reserves KV blocks for their whole max_seq.
 * Per layer i (App. I): the still-active tokens run layer i; for 2 <= i <= N-1 each
 * active token tests <s_hat_i, I_hat> >= delta (Sec. 4.1), or, where
 * d_forced_exit[j] != 0, exits exactly at that layer; exiting tokens are mapped by
 * the HSM (Sec. 4.2) and their K/V for every skipped layer r > i* are produced
 * from s~_N (Sec. 4.3) before layer r's attention.
 *   d_tokens        [batch*prompt_len] int32 token ids, sequence-major
 *   delta           exit threshold (+inf: never exit)
 *   d_forced_exit   [batch*prompt_len] int32, 0 = use delta, else i* in [2, N]; or NULL
 *   d_exit_layer_out[batch*prompt_len] int32 i* per token (N = full depth); or NULL
 *   d_logits_out    decoder: [batch, vocab] fp32 logits of each sequence's last token;
 *                   encoder: [batch, n_classes] classifier logits of position 0; or NULL
 *   d_next_token_out[batch] int32 greedy argmax of the logits (lowest index on ties); or NULL
 *   d_sim_out       [batch*prompt_len, N] fp32 cosine at each tested layer, NaN elsewhere; or NULL
 * Errors: INVALID_ARG, CAPACITY (batch > max_batch, prompt_len > max_seq). */
ADEPT_API adept_status adept_prefill(adept_model* m, int batch, int prompt_len, const int32_t* d_tokens,
                           float delta, const int32_t* d_forced_exit, int32_t* d_exit_layer_out,
                           float* d_logits_out, int32_t* d_next_token_out, float* d_sim_out,
                           void* stream);

/* One generation step (App. I, generation phase): token b of sequence b is appended
 * at that sequence's next position and exits independently of the others.  Same
 * per-token outputs as adept_prefill with batch rows.  Decoder families only.
 * Errors: INVALID_ARG, CAPACITY (a sequence is full). */
ADEPT_API adept_status adept_decode_step(adept_model* m, int batch, const int32_t* d_tokens, float delta,
                               const int32_t* d_forced_exit, int32_t* d_exit_layer_out,
                               float* d_logits_out, int32_t* d_next_token_out, float* d_sim_out,
                               void* stream);

/* Threshold calibration (Sec. 4.1: delta is set to meet the computation budget; Sec. 5.1):
 * bisection on delta in [lo, hi] over prompt passes of the calibration batch d_tokens
 * [batch, prompt_len] (threshold exits, no forced exits) until the batch's reduction in
 * computation RDC = 1 - sum(exit layer) / (batch prompt_len N) is within tol of target_rdc,
 * or max_iter passes have run.  A pass whose RDC is above the target raises the
 * threshold (lo = delta), otherwise it lowers it (hi = delta).
 *   delta_out, rdc_out, iters_out: host pointers (the last pass's delta and RDC, passes run)
 * Synchronous: waits for each pass on `stream`.  Like adept_prefill it resets sequences
 * 0..batch-1.  Errors: INVALID_ARG (target outside [0, 1), tol < 0, max_iter < 1,
 * lo >= hi, NULL pointers), and those of adept_prefill. */
ADEPT_API adept_status adept_calibrate_threshold(adept_model* m, int batch, int prompt_len, const int32_t* d_tokens,
                                       float target_rdc, float tol, int max_iter, float lo, float hi,
                                       float* delta_out, float* rdc_out, int* iters_out, void* stream);

/* Decoupled skipped-layer KV fill (Eq. 6, the decoupling of Sec. 4; Eq. 9, KV
 * generation in Sec. 4.3): for every token j and every layer r = i*_j+1..N, writes layer r's
 * K = RoPE(W_K^r norm_r(s~_j) + b_K^r) and V = W_V^r norm_r(s~_j) + b_V^r into the
 * KV cache at (d_seq[j], d_pos[j]); all (token, layer) pairs in one grouped launch.
 *   d_h_mapped  [n_tokens, D] mapped states s~_N in the model dtype
 *   d_exit_layer[n_tokens] int32 i* in [1, N] (N: nothing to fill)
 *   d_seq, d_pos[n_tokens] int32 sequence and position; their KV blocks must have been
 *               reserved (adept_prefill or adept_seq_reserve)
 * Errors: INVALID_ARG, CAPACITY (n_tokens above the fill workspace limit, 1<<20). */
ADEPT_API adept_status adept_skip_kv_fill(adept_model* m, int n_tokens, const void* d_h_mapped,
                                const int32_t* d_exit_layer, const int32_t* d_seq,
                                const int32_t* d_pos, void* stream);

/* Allocation-free variant of adept_skip_kv_fill.  The paper has no counterpart: this is
 * an interface for callers that cannot allocate device memory -- code recording a CUDA
 * graph (allocation and the synchronisation of cudaFree cannot be captured), serving
 * loops under a fixed memory budget or their own allocator, and latency-critical paths
 * that must not synchronise the device.  adept_skip_kv_fill grows a per-model workspace
 * with cudaMalloc when a call brings more tokens than before; this call keeps the same
 * working set in a fixed file-scope device array of ADEPT_NOALLOC_SCRATCH_BYTES bytes
 * (16 MiB, held by every GPU that loads the library until the process exits) and calls
 * no cudaMalloc, cudaFree or other allocating routine.  Same arguments and results as
 * adept_skip_kv_fill; bf16 models only.
 *  - Limit: n_tokens * (d_model * 2 + 4) bytes plus about 3 KiB must fit the array
 *    (about 2000 tokens at d_model 4096, 10900 at d_model 768); larger calls return
 *    ADEPT_ERR_CAPACITY with the limit in adept_last_error and enqueue nothing.
 *  - The first call on a device looks up the array's device address (with that device
 *    current); make that first call before any stream capture.
 *  - Every call shares the array and it keeps the last call's contents (each call clears
 *    the counters it needs zeroed).  Calls that overlap on the GPU -- on different streams
 *    or for different models on one device -- race on it: serialise them.
 *  - On the host the call keeps its launch description on the calling thread's stack and
 *    in thread-local storage: host threads that drive different models (on different
 *    devices, or one after the other on the GPU of one device) do not share host state.
 *    The calling thread's programmatic-dependent-launch setting is restored on return. */
#define ADEPT_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)
ADEPT_API adept_status adept_skip_kv_fill_noalloc(adept_model* m, int n_tokens, const void* d_h_mapped,
                                                  const int32_t* d_exit_layer, const int32_t* d_seq,
                                                  const int32_t* d_pos, void* stream);

/* Release everything the model owns (synchronises the device first).  NULL is a no-op. */
ADEPT_API void adept_free(adept_model* m);

/* Encoder-decoder models (Sec. 5.2, the OFA setting: an early-exiting encoder whose final
 * states feed a decoder that exits token by token too).  For a decoder loaded with
 * max_src > 0: set the source of every layer's cross-attention for sequences 0..n_seq-1.
 * d_states: fp32 [sum_b h_src_len[b]][d_model], device, in sequence order -- the encoder's
 * final states (s_N of tokens that ran to full depth, s~_N of exited ones; for an encoder
 * pass of n_seq x P tokens, the rows adept_read_final_states returns, with h_src_len[b] = P).
 * h_src_len[b] in [1, max_src].  Computes each decoder layer's source K/V (its cross K/V
 * projection of the states, rounded to bf16 for bf16 models) into the model's source cache;
 * later prompt passes and generation steps of these sequences cross-attend over all
 * h_src_len[b] source positions (not causal).  The states may be released once `stream` has
 * passed the call.  Errors: INVALID_ARG (no cross-attention, n_seq or a length out of range,
 * NULL pointer), CUDA. */
ADEPT_API adept_status adept_set_cross_source(adept_model* m, int n_seq, const int32_t* h_src_len,
                                              const float* d_states, void* stream);

/* ---- helpers (not part of the method; used by tests and the benchmark) ---- */

/* Message of the last failing call on `m` (or of the last failed load when m is NULL). */
ADEPT_API const char* adept_last_error(const adept_model* m);
ADEPT_API const char* adept_status_string(adept_status s);

/* Reset sequences 0..batch-1 to lengths h_lens[b] and reserve their KV blocks for
 * max_seq positions (no compute; the cached values are left undefined). */
ADEPT_API adept_status adept_seq_reserve(adept_model* m, int batch, const int32_t* h_lens);

/* Copy K and V of `n_pos` positions starting at pos0 of sequence `seq` at layer
 * `layer` (1-based) out of the paged cache into d_k_out / d_v_out, each
 * [n_pos, n_kv_heads, head_dim] in the model dtype. */
ADEPT_API adept_status adept_read_kv(adept_model* m, int layer, int seq, int pos0, int n_pos,
                           void* d_k_out, void* d_v_out, void* stream);

/* Copy the final states of the last prefill/decode pass ([rows, D] fp32: s~_N of
 * exited tokens, s_N of the rest) into d_out; rows = tokens of that pass. */
ADEPT_API adept_status adept_read_final_states(adept_model* m, float* d_out, int rows, void* stream);

/* Synchronise `stream`, then read and clear the device error word.
 * Returns DEVICE_INPUT if a kernel flagged an invalid input, TIMEOUT if a bounded
 * wait gave up, CUDA on an asynchronous CUDA error, else OK. */
ADEPT_API adept_status adept_check_device_status(adept_model* m, void* stream);

/* Options (ADEPT_OPT_*).  HSM_IDENTITY=1 replaces the HSM by s~ = s_i* (test switch).
 * PROFILE=1 records CUDA events around the GEMM, fill and attention launches so that
 * adept_profile_read can report launch counts and device time per kernel class
 * (generation steps then run as direct launches).  GEMM_SIMT=1 routes GEMMs to the
 * SIMT kernels (cross-check).  DECODE_GRAPH (default 1): from its second call with a
 * given batch size, adept_decode_step replays a CUDA graph of the step captured once;
 * 0 launches every kernel directly.  DECODE_GEMM (default 1): single GEMMs of at most 16
 * rows (generation steps, output heads) of bf16 models run on the weight-streaming
 * generation-step kernel, with the input standardisation fused in; 0 routes them to the
 * tcgen05 kernel after a separate standardisation launch.  DECODE_STREAM (default 1): those
 * weight-streaming GEMMs that are wide (at least 8192 outputs, or a grouped fill) and large
 * enough to stream (at least 8 MB of weights), and whose rows fit in shared memory, run on the
 * stream-K kernel (equal shares of the weight stream per SM, split tiles finished by the last
 * CTA to arrive); 0 keeps every one of them on the cluster K-split kernel.  DECODE_TILED (default 1): bf16 decoders keep a tile-contiguous copy of every streamed
 * weight (layer projections, LM head, the mapper's FC weights; made at load, refreshed after
 * each mapper training step; it doubles the weights' device memory) from which the weight-
 * streaming kernels fetch each 32-row x 256-k unit with one contiguous bulk copy; 0 makes them
 * read the row-major weights through tensor maps instead.  EXIT_METRIC (App. H.3): 0 (default) the global similarity of Sec. 4.1,
 * cos(s_i, sum_{d<i} s_hat_d); 1 the local similarity cos(s_i, s_{i-1}); 2 both (a token leaves
 * when both reach delta; the reported similarity is their minimum).  ALL_AT_ONCE (App. H.2):
 * 1 makes every token of a prompt take the exit decision of its sequence's last prompt token,
 * so a sequence leaves at once (generation steps are unaffected: one token per sequence).
 * Default 0.  STOP_ENTIRELY (bf16 encoders; Sec. 4.3 on downstream tasks): 1 stops an exited
 * token's computation entirely — no K/V of deeper layers, and deeper layers' attention sees
 * only the tokens still active there; its mapped state still feeds the classifier.  Default 0.
 * SPAN_TIMER (instrumentation, default 0): 1 makes the weight-streaming GEMM launches (the
 * stream-K and the cluster K-split kernel: generation steps, output heads of short passes,
 * fills of a few tokens) record their span on the device timer, from the first CTA past the
 * grid-dependency wait to the end of the last CTA, summed per kernel class by a small kernel at
 * the end of each pass (read with adept_span_read; a pass records its first 1024 such launches).
 * Launches keep programmatic dependent launch and graph replay (graphs are captured again),
 * so spans are taken in the step as it runs; consecutive launches' spans do not overlap.
 * ATTN_TC (default 1): the prompt-pass attention of bf16 models (self- and cross-attention,
 * head_dim 64 or 128) runs on the tcgen05 kernel (S and O accumulated in tensor memory, P
 * rounded to bf16); 0 keeps the mma.sync kernel (which the encoder's stop-entirely variant
 * always uses).  FUSED_EXIT (default 1): in generation steps of at most 4 sequences whose QKV
 * product runs on the stream-K kernel (decoders without cross-attention, global exit
 * similarity), the exit step of layer i (test, inertia update, compaction) is taken by layer
 * i+1's QKV launch: every CTA reduces the layer's rows and takes the same decisions, so the
 * separate exit kernel and its launch leave the step; 0 launches the exit kernel after every
 * layer. */
enum { ADEPT_OPT_HSM_IDENTITY = 1, ADEPT_OPT_PROFILE = 2, ADEPT_OPT_GEMM_SIMT = 3, ADEPT_OPT_DECODE_GRAPH = 4,
       ADEPT_OPT_DECODE_GEMM = 5, ADEPT_OPT_EXIT_METRIC = 7, ADEPT_OPT_ALL_AT_ONCE = 8,
       ADEPT_OPT_STOP_ENTIRELY = 9, ADEPT_OPT_DECODE_STREAM = 10, ADEPT_OPT_DECODE_TILED = 11,
       ADEPT_OPT_SPAN_TIMER = 12, ADEPT_OPT_ATTN_TC = 13, ADEPT_OPT_FUSED_EXIT = 14 };
ADEPT_API adept_status adept_set_option(adept_model* m, int option, int value);

/* Kernel classes reported by adept_profile_read: the GEMMs of prompt passes (layer
 * projections, HSM, head, and the per-layer skipped-layer fills co-launched with
 * layer i's QKV), the GEMMs of generation steps, the grouped skipped-layer fill
 * launches (end of a generation step and adept_skip_kv_fill), attention, and the GEMMs
 * of HSM training steps. */
enum { ADEPT_PROF_GEMM_PREFILL = 0, ADEPT_PROF_KV_FILL = 1, ADEPT_PROF_ATTENTION = 2,
       ADEPT_PROF_GEMM_DECODE = 3, ADEPT_PROF_GEMM_TRAIN = 4, ADEPT_PROF_NCLASS = 5 };
/* Synchronise, then return the number of recorded launches of kernel class `cls` and
 * their total device time in ms (CUDA events on the launching stream); resets the
 * record.  flops / bytes are reserved (returned as 0). */
ADEPT_API adept_status adept_profile_read(adept_model* m, int cls, int64_t* launches, double* total_ms,
                                double* flops, double* bytes);
/* Synchronise, then return the launches of class `cls` recorded by the span timer and their
 * summed spans in ms; resets the class total.  Zeros when the timer was never on. */
ADEPT_API adept_status adept_span_read(adept_model* m, int cls, int64_t* launches, double* total_ms);

/* ---- HSM training (Sec. 4.2; Sec. 4.3; Sec. 5.1 "Training"; App. D) -------------------
 * The Hidden State Mapper is trained with the base model frozen.  Decoders: its mapped state
 * s~ of an example (s_i, s_{i-1}, I) goes through the frozen final norm and LM head, and the
 * mean cross-entropy against the example's target token (the next input token) is minimised
 * (adept_hsm_train_step).  Encoders: a similarity loss against the original final hidden
 * states plus the frozen classifier's cross-entropy on the labelled rows
 * (adept_hsm_train_step_cls).  Both with AdamW (decoupled weight decay, bias-corrected
 * moments).
 *
 * Parameters, in this order (Table S1): 0 g0 [D], 1 conv_w [3][3], 2 conv_b [1], 3 fc1_w
 * [m1][D], 4 fc1_b [m1], 5 fc2_w [m2][m1], 6 fc2_b [m2], 7 fc3_w [m1][m2], 8 fc3_b [m1], 9 g1
 * [m1], 10 fc4_w [D][m1], 11 fc4_b [D], 12 g2 [D].  The library keeps fp32 master copies and
 * the two AdamW moments of each; the products run on the model dtype's GEMMs (bf16 models:
 * bf16 operands, fp32 accumulation), everything else in fp32.  After every step the model's
 * own HSM weights (used by adept_prefill / adept_decode_step) hold the updated values. */
typedef struct {
  float lr, beta1, beta2, eps, weight_decay;
} adept_adamw;

/* Starts HSM training: master parameters from the model's current HSM weights, zero moments,
 * step count 0, and device workspaces for up to max_rows examples per step (a second call
 * frees the previous ones and starts over).  Synchronous on `stream`.
 * Errors: INVALID_ARG (max_rows < 1, an encoder whose n_classes is outside [1, 64], a bf16
 * model whose D, m1 or m2 is not a multiple of 8), OOM. */
ADEPT_API adept_status adept_hsm_train_init(adept_model* m, int max_rows, void* stream);

/* One training step on n examples, enqueued on `stream`: forward (Table S1) with the
 * activations kept, frozen head, cross-entropy, backward, AdamW with step number t = (steps
 * so far) + 1, write-back of the model's HSM weights.
 *   d_s_i, d_s_prev, d_inertia  [n, D] fp32 device rows: s_i, s_{i-1} and I of each example
 *   d_target                    [n] int32 device token ids in [0, vocab) (a bad id flags
 *                               DEVICE_INPUT at adept_check_device_status; its row adds
 *                               nothing to the loss or the gradients)
 *   hp                          host pointer to the hyperparameters
 *   d_loss_out                  device float: the mean loss before the update (NULL: not written)
 * Errors: INVALID_ARG (no adept_hsm_train_init, an encoder model, n outside [1, max_rows],
 * NULL pointers, lr < 0, beta outside [0, 1), eps <= 0, weight_decay < 0). */
ADEPT_API adept_status adept_hsm_train_step(adept_model* m, int n, const float* d_s_i, const float* d_s_prev,
                                  const float* d_inertia, const int32_t* d_target, const adept_adamw* hp,
                                  float* d_loss_out, void* stream);

/* One training step of an encoder's HSM for classification (Sec. 4.3), enqueued on `stream`:
 * with no next token to predict, the loss is the similarity loss against the original final
 * hidden states, mean over the n examples of 1 - cos(s~, s_N) (cos = 0 where a norm is 0),
 * plus cls_weight times the frozen pooler + classifier's softmax cross-entropy (for two
 * classes, the binary cross-entropy) on the first n_cls examples, the labelled [CLS] rows,
 * averaged over them.  Then backward, AdamW and the weight write-back as adept_hsm_train_step.
 *   d_s_i, d_s_prev, d_inertia  [n, D] fp32 device rows as in adept_hsm_train_step
 *   d_s_final                   [n, D] fp32 device rows: the original final hidden states
 *   n_cls, d_label              labelled rows 0..n_cls-1 (0 <= n_cls <= n) and their int32 class
 *                               ids in [0, n_classes) on the device (NULL allowed when n_cls = 0;
 *                               a bad id flags DEVICE_INPUT at adept_check_device_status and its
 *                               row adds no task loss or gradient)
 *   cls_weight                  weight of the task loss (>= 0; the paper adds the two: 1)
 *   hp, d_loss_out              as in adept_hsm_train_step
 * Errors: INVALID_ARG (no adept_hsm_train_init, a decoder model, n or n_cls out of range, NULL
 * pointers, cls_weight < 0 or not finite, AdamW hyperparameters as above). */
ADEPT_API adept_status adept_hsm_train_step_cls(adept_model* m, int n, const float* d_s_i, const float* d_s_prev,
                                      const float* d_inertia, const float* d_s_final, int n_cls,
                                      const int32_t* d_label, float cls_weight, const adept_adamw* hp,
                                      float* d_loss_out, void* stream);

/* Copies one parameter's fp32 training values to device memory d_out (count = its element
 * count, adept_hsm_param_numel): what = ADEPT_HSM_PARAMS (master values), ADEPT_HSM_GRADS
 * (gradients of the last step), ADEPT_HSM_MOMENT1 / ADEPT_HSM_MOMENT2 (AdamW moments).
 * Enqueued on `stream`.  Errors: INVALID_ARG (no training state, bad what / param / count). */
enum { ADEPT_HSM_PARAMS = 0, ADEPT_HSM_GRADS = 1, ADEPT_HSM_MOMENT1 = 2, ADEPT_HSM_MOMENT2 = 3 };
ADEPT_API adept_status adept_hsm_train_read(adept_model* m, int what, int param, float* d_out, int64_t count,
                                  void* stream);
/* Element count of HSM parameter `param` (0..12), or -1. */
ADEPT_API int64_t adept_hsm_param_numel(const adept_model* m, int param);

/* ---- failure injection (tests of the error paths; no GPU fault is involved) ------------
 * adept_set_wait_limit: limit, in SM cycles, of the kernels' bounded waits on pipeline
 * progress (a ring slot being filled or released, an accumulator becoming ready) in the
 * tensor-core, weight-streaming and stream-K GEMMs; 0 restores the default (4e9 cycles, about
 * 2 s).  A wait that runs out sets the device error word, its CTA stops, lets the copies it
 * has in flight land (those waits, and the waits of cross-CTA reductions, keep their own long
 * limits), frees its tensor memory and exits, and adept_check_device_status then returns
 * ADEPT_ERR_TIMEOUT; the outputs of that call are undefined and the model stays usable.
 * Applies to every model of the process on the current device.  Errors: INVALID_ARG
 * (cycles < 0), CUDA.
 * adept_set_alloc_fail_after: after n more device allocations by the library, every further
 * allocation fails as if the device were out of memory (n < 0: off, the default); calls that
 * need memory then return ADEPT_ERR_OOM with everything they allocated released. */
ADEPT_API adept_status adept_set_wait_limit(int64_t cycles);
ADEPT_API void adept_set_alloc_fail_after(int64_t n);

/* Number of kernel launches the library enqueued since the last call (then reset). */
ADEPT_API int64_t adept_launch_count(adept_model* m);

#ifdef __cplusplus
}
#endif
#endif /* ADEPT_H */

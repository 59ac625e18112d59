/*
 * libbuddy — budget-routed batched decode (BUDDY, arXiv 2606.09514) on one
 * NVIDIA GB300 (sm_103a).
 *
 * One decode step, for every sequence i of a batch:
 *   1. runs the first decoder block (always executed, Sec. 4.2.1) -- blocks
 *      0..c with a context layer c > 0 (App. D, Start Layer ablation);
 *   2. pools the context layer's cache (value states by default, or key states,
 *      or their sum, Sec. 5.4), including the newest token, and concatenates
 *      the newest token's hidden state (KV-aware planner, Sec. 4.3);
 *   3. scores the routed blocks c+1 .. L-2 with the Decision Module, a
 *      Linear-SiLU-Linear MLP (App. C.1), fused with an optional prior
 *      s' = s + omega * p~ (Eq. 2); a sequence without a budget (k_i = 0)
 *      takes the Budget Predictor's k^ (Sec. 4.4);
 *   4. executes the k_i highest-scoring routed blocks (Eq. 2, ties to the lower
 *      layer index), each block on the sub-batch of sequences that selected it
 *      (grouping by mask, App. C.1), skipped blocks being the identity (Eq. 1)
 *      and storing zero K/V at the new position (Sec. 6) -- or nothing, in the
 *      masked variant;
 *   5. runs the last block (always executed) and advances every sequence's
 *      position by one (KV cache update, Eq. 9).
 *
 * buddy_prefill does the same for whole prompts: one route per prompt, every
 * prompt token through the selected blocks (Sec. 4.1, App. E).
 *
 * Conventions for every entry point:
 *   - Pointers marked "device" are device pointers owned by the caller; the
 *     library never frees them.  Weight pointers are retained (not copied) by
 *     buddy_set_weights and must stay valid while the context is used.
 *   - Weight matrices and norm gains, the K/V caches, the pooled sums and the
 *     hidden-state buffers (h_in, h_out, prefill x, route h1) must be 16-byte
 *     aligned (the kernels access them with 16-byte vectors and TMA); a
 *     misaligned one is rejected with BUDDY_ERR_ARG.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Calls are asynchronous on that stream unless stated otherwise.
 *   - Return value: BUDDY_OK or a BUDDY_ERR_* code.  On a host-detected error
 *     nothing is launched and nothing is written.  Conditions that only the
 *     device can see (a budget or position stored in device memory out of
 *     range) make every kernel of that call return without writing; the flag
 *     is reported by buddy_device_status().
 *   - The library allocates device memory only in buddy_create (scratch sized
 *     by max_batch, max_pos and max_prefill_tokens), in buddy_set_weights
 *     (tensor descriptors, split-K workspace) and in
 *     buddy_set_budget_predictor (its hidden units).
 */
#ifndef BUDDY_H_
#define BUDDY_H_

#include <stdint.h>

#if defined(__GNUC__)
#define BUDDY_API __attribute__((visibility("default")))
#else
#define BUDDY_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

enum {
  BUDDY_OK = 0,
  BUDDY_ERR_ARG = 1,      /* null pointer, bad size, unsupported shape */
  BUDDY_ERR_RANGE = 2,    /* value outside its documented range (host-visible) */
  BUDDY_ERR_CUDA = 3,     /* a CUDA runtime call failed */
  BUDDY_ERR_DEVICE = 4,   /* a kernel raised the device error flag */
  BUDDY_ERR_STATE = 5     /* call order: e.g. weights not set */
};

enum { BUDDY_DTYPE_F32 = 0, BUDDY_DTYPE_BF16 = 1 };

/* Planner feature G_t pooled from the context layer's cache (Sec. 4.3; the
 * Sec. 5.4 ablation "Hidden-State Features"): value states (the paper's
 * default), key states (as cached, after RoPE), or their element-wise sum. */
enum { BUDDY_FEATURE_V = 0, BUDDY_FEATURE_K = 1, BUDDY_FEATURE_KV = 2 };

/* KV of a sequence at a block it skips (Sec. 6): zero-filled K and V at the
 * new position, which later attention includes with logit 0 (the paper's
 * design); or nothing stored, so that block's later attention reads only the
 * positions at which it executed (the KV-cache strategy Sec. 6 leaves to
 * future work). */
enum { BUDDY_SKIP_ZERO = 0, BUDDY_SKIP_MASKED = 1 };

/* Bits of the device error flag (buddy_device_status). */
enum {
  BUDDY_DEV_BAD_BUDGET = 1,    /* k_i outside [1, L-2-c] (0 without a Budget Predictor) */
  BUDDY_DEV_BAD_POSITION = 2,  /* len_i + new positions > cap_i or > max_pos */
  BUDDY_DEV_BAD_SEQ = 4,       /* a sequence id outside [0, batch) */
  BUDDY_DEV_TIMEOUT = 8        /* a bounded wait inside a kernel ran out */
};

typedef struct buddy_ctx buddy_ctx;

/* Model shape.  The decoder block is Llama-style (App. "Background"):
 * RMSNorm, Q/K/V projections (optional bias, Qwen2.5), rotate-half RoPE,
 * grouped-query attention, output projection, RMSNorm, SwiGLU MLP d->F->d.
 * Requirements: n_layers >= 3; head_dim 64 or 128; n_q_heads a multiple of
 * n_kv_heads (group of at most 8); d_model == n_q_heads * head_dim, a
 * multiple of 64; ffn_dim a multiple of 8; dm_hidden >= 1;
 * 1 <= max_batch <= 1024 (<= 256 for bf16, which needs an sm_103 device);
 * max_pos >= 1; 0 <= ctx_layer <= n_layers - 3; 0 <= max_prefill_tokens
 * <= 65536.  The routed blocks are ctx_layer+1 .. n_layers-2: their number
 * n_cand = n_layers - 2 - ctx_layer sizes the Decision Module's output. */
typedef struct {
  int32_t n_layers;     /* L */
  int32_t d_model;      /* d */
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t ffn_dim;      /* F */
  int32_t dm_hidden;    /* r: Decision Module hidden width */
  int32_t dtype;        /* BUDDY_DTYPE_F32 or BUDDY_DTYPE_BF16: weights, KV cache, GEMM inputs */
  int32_t max_batch;    /* largest B of any call */
  int32_t max_pos;      /* every position p written or read satisfies p < max_pos */
  int32_t qkv_bias;     /* 1: Q/K/V projections carry a bias */
  int32_t feature;      /* BUDDY_FEATURE_*: planner feature */
  int32_t ctx_layer;    /* c: blocks 0..c always run, the planner reads block c's cache */
  int32_t skip_kv;      /* BUDDY_SKIP_*: what a skipped block stores */
  int32_t max_prefill_tokens;  /* 0: no buddy_prefill; else the largest sum of prompt lengths */
  float rms_eps;
  float rope_theta;
} buddy_config;

/* One decoder layer; matrices row-major in nn.Linear layout [out, in],
 * element type = config dtype; gains and biases fp32. */
typedef struct {
  const float* attn_norm;   /* device [d] */
  const void* w_qkv;        /* device [(n_q + 2 n_kv) * hd, d]: Q rows, then K rows, then V rows */
  const float* b_qkv;       /* device [(n_q + 2 n_kv) * hd], or NULL when qkv_bias == 0 */
  const void* w_o;          /* device [d, n_q * hd] */
  const float* ffn_norm;    /* device [d] */
  const void* w_gate_up;    /* device [2F, d]: rows [0, F) gate, rows [F, 2F) up */
  const void* w_down;       /* device [d, F] */
} buddy_layer_weights;

/* Decision Module (App. C.1): s' = W2 SiLU(W1 x + b1) + b2 + omega * prior,
 * x = [pool expanded to d ; h] of width 2d (Sec. 4.3).  All fp32.
 * n_cand = n_layers - 2 - ctx_layer. */
typedef struct {
  const float* w1;      /* device [r, 2d] */
  const float* b1;      /* device [r] */
  const float* w2;      /* device [n_cand, r] */
  const float* b2;      /* device [n_cand] */
  const float* prior;   /* device [n_cand] normalised prior p~ (Eq. 2), or NULL */
  float omega;          /* prior weight (ignored when prior == NULL) */
} buddy_dm_weights;

/* Budget Predictor (Sec. 4.4): a categorical policy pi(k | G_t) over
 * A = {1..n_cand} on the Decision Module's input x, here the same
 * Linear-SiLU-Linear form: logits = W2 SiLU(W1 x + b1) + b2; k^ = argmax
 * (ties to the smaller k), i.e. budget b^ = (k^ + 2 + ctx_layer) / L (Eq. 3).
 * All fp32. */
typedef struct {
  const float* w1;      /* device [hidden, 2d] */
  const float* b1;      /* device [hidden] */
  const float* w2;      /* device [n_cand, hidden] */
  const float* b2;      /* device [n_cand] */
  int32_t hidden;       /* >= 1 */
} buddy_predictor_weights;

/* Per-layer KV caches and per-sequence positions (Eq. 9).
 * Element (sequence i, kv head g, position p, channel e) of layer l's K cache
 * is at  k_cache[l] + ((seq_off[i] * n_kv + g * cap[i] + p) * head_dim + e)
 * elements (same for V): each sequence owns a head-major block of cap[i]
 * positions; blocks must not overlap.  len[i] = tokens n_i of sequence i (the
 * RoPE position of its next token).  With BUDDY_SKIP_ZERO every layer holds
 * len[i] cached positions; with BUDDY_SKIP_MASKED layer l holds
 * layer_len[l * batch + i] <= len[i] (the positions at which it executed).
 * pool_sum[i] = running fp32 sum over the context layer's cached positions of
 * the planner feature (the KV-aware planner's context, Sec. 4.3). */
typedef struct {
  void* const* k_cache;     /* host array [L] of device pointers (config dtype) */
  void* const* v_cache;     /* host array [L] of device pointers */
  const int64_t* seq_off;   /* device [batch] */
  const int32_t* cap;       /* device [batch] */
  int32_t* len;             /* device [batch] */
  float* pool_sum;          /* device [batch, n_kv * hd] */
  int32_t batch;            /* number of sequences the state holds */
  int32_t* layer_len;       /* device [L, batch] with BUDDY_SKIP_MASKED, else NULL */
} buddy_kv_state;

/* Creates a context on the current device; allocates its scratch. */
BUDDY_API int buddy_create(const buddy_config* cfg, buddy_ctx** out);
BUDDY_API void buddy_destroy(buddy_ctx* ctx);

/* Registers the model: layers[0..L-1] and the Decision Module.  Pointers are
 * retained.  Builds the TMA tensor descriptors of the bf16 weight matrices.
 * BUDDY_ERR_ARG for a bf16 context the tensor-core path cannot serve (a
 * device other than sm_103). */
BUDDY_API int buddy_set_weights(buddy_ctx* ctx, const buddy_layer_weights* layers, const buddy_dm_weights* dm);

/* Registers (bp != NULL) or removes (NULL) the Budget Predictor (Sec. 4.4).
 * With one registered, a budget k_i = 0 in buddy_decode_step, buddy_route or
 * buddy_prefill means "no budget given": the sequence executes the
 * predictor's k^ routed blocks.  Pointers are retained.  Allocates the
 * predictor's hidden units (max_batch * hidden fp32). */
BUDDY_API int buddy_set_budget_predictor(buddy_ctx* ctx, const buddy_predictor_weights* bp);

/* Bulk append of n_new given positions to layer `layer` for n_seq sequences
 * (KV cache update, Eq. 9), e.g. to load a prefilled cache.  k_new, v_new:
 * device [n_seq, n_new, n_kv, hd] (config dtype), written at positions
 * p0 .. p0 + n_new - 1 of sequence s = seq_ids[j], p0 = len[s]
 * (BUDDY_SKIP_MASKED: p0 = layer_len[layer][s], which then grows by n_new).
 * For the context layer the pooled context pool_sum[s] is recomputed as the
 * full sum of the planner feature over positions 0 .. p0 + n_new - 1.
 * advance != 0 adds n_new to len[s] afterwards (pass it on the last layer
 * appended).  seq_ids must be distinct.  Device-checked: s < kv->batch,
 * p0 + n_new <= cap[s] and <= max_pos. */
BUDDY_API int buddy_kv_append(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t layer, int32_t n_seq,
                    const int32_t* seq_ids, int32_t n_new, const void* k_new, const void* v_new,
                    int32_t advance, void* stream);

/* The router alone (KV-aware planner + Decision Module + top-k, Sec. 4.2-4.3):
 * for i < batch, pool = pool_sum[i] / len[i] (the cache must already hold the
 * newest token at position len[i]-1), x = [pool expanded; h1[i]],
 * s' as in buddy_dm_weights, selection = the k[i] largest s' (ties to the lower
 * index; k[i] = 0: the Budget Predictor's k^).  h1: device [batch, d] fp32,
 * the newest token's state after block c; k: device [batch] int32 in
 * [1, n_cand] (or 0).  Outputs (device, any may be NULL): sel_out
 * [batch, n_cand] int32 — executed layer ids (c+1..L-2, ascending) then -1;
 * mask_out [batch, L] uint8 (blocks 0..c and the last set); scores_out
 * [batch, n_cand] fp32. */
BUDDY_API int buddy_route(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch, const float* h1,
                const int32_t* k, int32_t* sel_out, uint8_t* mask_out, float* scores_out,
                void* stream);

/* Allocation-free router, for callers that cannot allocate device memory and
 * therefore cannot create a buddy_ctx: for example a process whose device
 * memory is all owned by its own pool allocator, or code that runs where
 * cudaMalloc (which may synchronise the device) is not allowed.  The paper
 * has no counterpart; this is a deployment variant of buddy_route.
 *
 * Computes what buddy_route computes for a context with ctx_layer 0 and no
 * Budget Predictor, from explicit arguments instead of a context: shape
 * (n_layers, d_model, n_q_heads, n_kv_heads, head_dim, dm_hidden, same rules
 * as buddy_config), Decision Module `dm` (n_cand = n_layers - 2), and device
 * arrays pool_sum [batch, n_kv*hd], len [batch] (>= 1, the cache already holds
 * the newest token), h1 [batch, d] fp32, k [batch].  Outputs as buddy_route;
 * flags_out (device int32, may be NULL) receives the BUDDY_DEV_* bits of this
 * call (0 when valid; on a nonzero value nothing else was written).
 *
 * Scratch: one static device array of the library (256 KiB of hidden units
 * plus a small header), held by every GPU that loads the library until the
 * process exits.  batch * dm_hidden must not exceed 65536, else
 * BUDDY_ERR_RANGE.  The first call on each device looks up the array's
 * device address (cudaGetSymbolAddress); make that first call outside any
 * stream capture.  The address is cached for the life of the process: after
 * cudaDeviceReset (or anything else that recreates the device's primary
 * context) the library must be reloaded before this entry is called again.
 * All calls share the array: calls whose kernels overlap on the GPU
 * (different streams without ordering) race.  Allocates nothing. */
BUDDY_API int buddy_route_noalloc(int32_t n_layers, int32_t d_model, int32_t n_q_heads,
                                  int32_t n_kv_heads, int32_t head_dim, int32_t dm_hidden,
                                  const buddy_dm_weights* dm, int32_t batch, const float* pool_sum,
                                  const int32_t* len, const float* h1, const int32_t* k,
                                  int32_t* sel_out, uint8_t* mask_out, float* scores_out,
                                  int32_t* flags_out, void* stream);

/* One budget-routed decode step for sequences 0..batch-1 of `kv`.
 * h_in: device [batch, d] fp32 (input of the first block); k: device [batch]
 * int32 budgets in [1, n_cand] (0: predicted); h_out: device [batch, d] fp32,
 * the hidden state after the last block (must not alias h_in).  Optional
 * device outputs (NULL to skip): mask_out [batch, L] uint8; rows_out [L,
 * batch] int32 (for layer l the ascending ids of the sequences that execute
 * it, then unspecified); count_out [L] int32 (their number); scores_out
 * [batch, n_cand] fp32.  Every layer's cache receives one position per
 * sequence (zeros for skipped layers; with BUDDY_SKIP_MASKED only executed
 * layers store one, and layer_len counts them) and len[i] += 1.
 * Device-checked: k[i] in range, len[i] + 1 <= cap[i] and <= max_pos, and
 * with BUDDY_SKIP_MASKED 0 <= layer_len[l][i] <= len[i]; on failure nothing is
 * written. */
BUDDY_API int buddy_decode_step(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch, const float* h_in,
                      const int32_t* k, float* h_out, uint8_t* mask_out, int32_t* rows_out,
                      int32_t* count_out, float* scores_out, void* stream);

/* Routed prefill of one prompt per sequence (Sec. 4.1; App. E "Prefill vs.
 * Decode"), bf16 contexts created with max_prefill_tokens > 0.
 * n_tok: HOST [batch] prompt lengths (>= 1, sum <= max_prefill_tokens);
 * x: device [sum n_tok, d] fp32, the prompts' input hidden states, sequence
 * by sequence (rows off_i .. off_i + n_tok[i] - 1 for sequence i, off_i the
 * sum of the earlier lengths); k: device [batch] budgets as in
 * buddy_decode_step; h_out: device [sum n_tok, d] fp32, every token's hidden
 * state after the last block (must not alias x).  Optional device outputs:
 * mask_out [batch, L] uint8, scores_out [batch, n_cand] fp32.
 * Sequence i's tokens take positions len[i] .. len[i] + n_tok[i] - 1.  Blocks
 * 0..c run on every token with causal attention; each sequence is routed once
 * from its pooled context-layer cache (prompt included) and its last token's
 * state after block c; each routed block runs on all tokens of the sequences
 * that selected it; a skipped block stores zero K/V at every prompt position
 * (BUDDY_SKIP_MASKED: nothing).  Then len[i] += n_tok[i].  The call
 * synchronises `stream` once, after the routing, to size the later launches;
 * it returns BUDDY_ERR_DEVICE (nothing written) when the device checks of
 * buddy_decode_step fail (budgets, len[i] + n_tok[i] <= cap[i], <= max_pos). */
BUDDY_API int buddy_prefill(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch, const int32_t* n_tok,
                            const float* x, const int32_t* k, float* h_out, uint8_t* mask_out,
                            float* scores_out, void* stream);

/* buddy_decode_step with HOST buffers: h_in_host [batch, d] fp32, k_host
 * [batch] int32, h_out_host [batch, d] fp32, mask_host [batch, L] uint8 (or
 * NULL).  Copies the inputs to device staging buffers, runs the step, copies
 * the outputs back and synchronises the stream before returning.  Pinned host
 * memory gives asynchronous copies; pageable memory works but is slower. */
BUDDY_API int buddy_decode_step_host(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch,
                           const float* h_in_host, const int32_t* k_host, float* h_out_host,
                           uint8_t* mask_host, void* stream);

/* Execution options.  use_graph != 0: buddy_decode_step replays a CUDA graph
 * of the step's launches, captured per (batch, kv state, stream) on first use;
 * the kernels of a layer that no sequence selected exit as soon as they start.
 * The graph bakes in the pointers of that call; a call with other pointers
 * re-captures. */
BUDDY_API int buddy_set_options(buddy_ctx* ctx, int32_t use_graph);

/* Which kernels a context runs (valid after buddy_set_weights), so that a
 * measurement can state them: paths[0] GEMM (0 CUDA-core fp32, 1 tcgen05
 * bf16), paths[1] attention (0 CUDA-core, 1 mma.sync tensor-core loop over
 * the whole GPU, 2 the same contractions with one thread-block cluster per
 * (row, KV head) stream, for small batches),
 * paths[2] RMSNorm computed inside the QKV and gate/up GEMMs (0/1),
 * paths[3] split-K sums in a separate fixup kernel (0/1).  n <= 4 entries. */
BUDDY_API int buddy_get_paths(buddy_ctx* ctx, int32_t* paths, int32_t n);

/* Limit of every bounded wait inside the tensor-core GEMM pipelines (TMA
 * stages, MMA completion, accumulator hand-over), in nanoseconds; ns <= 0
 * restores the default of 4 s.  A wait that runs out makes its kernel stop
 * (after its copies and MMAs in flight have completed), raise
 * BUDDY_DEV_TIMEOUT and leave its outputs incomplete; buddy_device_status
 * then reports the bit and re-arms the kernels' arrival counters, so the
 * context stays usable.  Synchronises the device; drops captured graphs. */
BUDDY_API int buddy_set_wait_limit(buddy_ctx* ctx, int64_t ns);

/* Kernel classes reported by the profiler. */
enum {
  BUDDY_PROF_CHECK = 0, BUDDY_PROF_RMSNORM, BUDDY_PROF_GEMM_QKV, BUDDY_PROF_QKV_FINALIZE,
  BUDDY_PROF_ATTENTION, BUDDY_PROF_GEMM_O, BUDDY_PROF_GEMM_GATE_UP, BUDDY_PROF_GEMM_DOWN,
  BUDDY_PROF_ROUTE, BUDDY_PROF_COMPACT, BUDDY_PROF_OTHER,
  BUDDY_PROF_GEMM_FIXUP,   /* split-K sums + epilogues of the GEMMs (larger batches) */
  BUDDY_PROF_PF_GEMM,      /* prefill: projections (tcgen05, M-tiled) */
  BUDDY_PROF_PF_ATTENTION, /* prefill: causal attention */
  BUDDY_PROF_PF_OTHER,     /* prefill: RMSNorm, zero fill, advance */
  BUDDY_PROF_NCLASS
};

/* Per-kernel-class timing.  With on != 0, direct-launch decode steps
 * (use_graph == 0) record a CUDA event pair on the launching stream around
 * every kernel launch, and count the launches.  buddy_profile_read
 * synchronises those events, writes per class the summed milliseconds and the
 * launch count (arrays of n_cls entries, n_cls <= BUDDY_PROF_NCLASS), and
 * clears the records.  buddy_profile_class_name gives a class's name. */
BUDDY_API int buddy_set_profiling(buddy_ctx* ctx, int32_t on);
BUDDY_API int buddy_profile_read(buddy_ctx* ctx, int32_t n_cls, float* ms, int32_t* launches);
BUDDY_API const char* buddy_profile_class_name(int32_t cls);

/* Synchronises `stream`, stores the device error flag bits (BUDDY_DEV_*) in
 * *flags and clears them.  Returns BUDDY_ERR_DEVICE if any bit was set. */
BUDDY_API int buddy_device_status(buddy_ctx* ctx, void* stream, int32_t* flags);

/* Budget b in (0, 1] to middle-layer count: k = round(b * L) - 2 (Eq. 2,
 * ties to even), clamped to the action space [1, L-2] (Sec. 4.4).
 * Returns -1 if n_layers < 3 or b is not finite. */
BUDDY_API int32_t buddy_budget_to_k(float b, int32_t n_layers);

BUDDY_API const char* buddy_error_string(int32_t code);
BUDDY_API int32_t buddy_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BUDDY_H_ */

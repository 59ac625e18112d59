// C-ABI of libbuddy: argument validation, scratch management, and the
// orchestration of one budget-routed decode step (direct launches or a CUDA
// graph of the same launches; layers no sequence selected exit at once).
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <new>
#include <tuple>

#include "../../include/buddy.h"
#include "internal.h"

using namespace buddy;

struct buddy_ctx {
  Ctx c;
  cudaStream_t cap_stream = nullptr;   // graph capture (the legacy stream cannot be captured)
};

#define CK(x)                                                     \
  do {                                                            \
    cudaError_t e_ = (x);                                         \
    if (e_ != cudaSuccess) {                                      \
      fprintf(stderr, "libbuddy: %s -> %s (%s:%d)\n", #x,         \
              cudaGetErrorString(e_), __FILE__, __LINE__);        \
      return BUDDY_ERR_CUDA;                                      \
    }                                                             \
  } while (0)

namespace buddy {
bool Ctx::GraphKey::operator<(const GraphKey& o) const {
  return std::tie(B, h_in, k, h_out, mask, rows, count, scores, stream, kvp) <
         std::tie(o.B, o.h_in, o.k, o.h_out, o.mask, o.rows, o.count, o.scores, o.stream, o.kvp);
}
int gemm_tc_prepare(Ctx& c);   // gemm_tc.cu
}  // namespace buddy

template <typename T>
static cudaError_t dalloc(T** p, size_t n) {
  *p = nullptr;
  if (n == 0) n = 1;
  return cudaMalloc((void**)p, n * sizeof(T));
}

static void free_ctx(buddy_ctx* x) {
  if (!x) return;
  Ctx& c = x->c;
  for (auto& kv : c.graphs) cudaGraphExecDestroy(kv.second);
  for (cudaEvent_t e : c.ev_pool) cudaEventDestroy(e);
  void* ptrs[] = {c.rope_cos, c.rope_sin, c.status, c.xn, c.act, c.attn_out, c.qkv, c.q,
                  c.attn_m, c.attn_l, c.attn_acc, c.attn_ctr, c.dm_u, c.dm_x, c.mask, c.sel, c.scores, c.rows,
                  c.count, c.h_in_stage, c.h_out_stage, c.k_stage, c.mask_stage, c.xn_lo, c.act_lo, c.attn_lo,
                  c.gemm_ws, c.gemm_ctr, c.pf_xn, c.pf_xn_lo, c.pf_q, c.pf_attn, c.pf_attn_lo,
                  c.pf_act, c.pf_act_lo, c.pf_tok_seq, c.pf_tok_t, c.pf_tok_pos, c.pf_rows, c.pf_items,
                  c.pf_n_tok, c.pf_tok_end, c.pf_cnt, c.pf_hlast};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  if (x->cap_stream) cudaStreamDestroy(x->cap_stream);
  delete x;
}

extern "C" int32_t buddy_version(void) { return 1; }

extern "C" const char* buddy_error_string(int32_t code) {
  switch (code) {
    case BUDDY_OK: return "ok";
    case BUDDY_ERR_ARG: return "invalid argument";
    case BUDDY_ERR_RANGE: return "value out of range";
    case BUDDY_ERR_CUDA: return "CUDA runtime error";
    case BUDDY_ERR_DEVICE: return "device error flag raised";
    case BUDDY_ERR_STATE: return "invalid call order (weights not set?)";
    default: return "unknown error";
  }
}

extern "C" int32_t buddy_budget_to_k(float b, int32_t n_layers) {
  if (n_layers < 3 || !std::isfinite(b)) return -1;
  // k = round(b L) - 2 with ties to even (Eq. 2), clamped to {1..L-2} (Sec. 4.4)
  const double k = std::nearbyint((double)b * (double)n_layers) - 2.0;
  const double lo = 1.0, hi = (double)(n_layers - 2);
  return (int32_t)(k < lo ? lo : (k > hi ? hi : k));
}

extern "C" int buddy_create(const buddy_config* cfg, buddy_ctx** out) {
  if (!cfg || !out) return BUDDY_ERR_ARG;
  *out = nullptr;
  const buddy_config& g = *cfg;
  if (g.n_layers < 3 || g.n_layers > kMaxLayers || g.d_model <= 0 || g.n_q_heads <= 0 ||
      g.n_kv_heads <= 0 || (g.head_dim != 64 && g.head_dim != 128) ||
      g.n_q_heads % g.n_kv_heads != 0 || g.n_q_heads / g.n_kv_heads > 8 ||
      g.d_model != g.n_q_heads * g.head_dim || g.d_model % 64 != 0 || g.ffn_dim <= 0 ||
      g.ffn_dim % 8 != 0 || g.dm_hidden <= 0 || g.max_batch < 1 || g.max_batch > kMaxBatch ||
      g.max_pos < 1 || (g.dtype != BUDDY_DTYPE_F32 && g.dtype != BUDDY_DTYPE_BF16) ||
      !(g.rms_eps > 0.f) || !(g.rope_theta > 0.f) ||
      (g.feature != BUDDY_FEATURE_V && g.feature != BUDDY_FEATURE_K && g.feature != BUDDY_FEATURE_KV) ||
      g.ctx_layer < 0 || g.ctx_layer > g.n_layers - 3 ||
      (g.skip_kv != BUDDY_SKIP_ZERO && g.skip_kv != BUDDY_SKIP_MASKED) || g.max_prefill_tokens < 0 ||
      g.max_prefill_tokens > 65536 || (g.dtype == BUDDY_DTYPE_BF16 && g.max_batch > 256))
    return BUDDY_ERR_ARG;
  buddy_ctx* x = new (std::nothrow) buddy_ctx();
  if (!x) return BUDDY_ERR_CUDA;
  Ctx& c = x->c;
  c.cfg = g;
  c.L = g.n_layers; c.cl = g.ctx_layer; c.Lm = g.n_layers - 2 - g.ctx_layer; c.d = g.d_model; c.nq = g.n_q_heads;
  c.feature = g.feature;
  c.masked = g.skip_kv == BUDDY_SKIP_MASKED;
  c.nkv = g.n_kv_heads; c.hd = g.head_dim; c.F = g.ffn_dim; c.r = g.dm_hidden;
  c.qd = c.nq * c.hd; c.kvd = c.nkv * c.hd; c.qkvN = c.qd + 2 * c.kvd;
  c.maxB = g.max_batch; c.max_pos = g.max_pos; c.dtype = g.dtype;
  c.esz = g.dtype == BUDDY_DTYPE_BF16 ? 2 : 4;
  auto fail = [&](cudaError_t e) {
    fprintf(stderr, "libbuddy: create: %s\n", cudaGetErrorString(e));
    free_ctx(x);
    return BUDDY_ERR_CUDA;
  };
  cudaError_t e;
  if ((e = cudaGetDevice(&c.device)) != cudaSuccess) return fail(e);
  if ((e = cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, c.device)) != cudaSuccess)
    return fail(e);
  const size_t B = c.maxB;
  c.attn_max_chunks = attention_max_spans(c.max_pos);
  const size_t hmax = (size_t)c.max_pos * (c.hd / 2);
  if ((e = dalloc(&c.rope_cos, hmax)) || (e = dalloc(&c.rope_sin, hmax)) ||
      (e = dalloc(&c.status, 4)) ||
      (e = cudaMalloc(&c.xn, B * c.d * c.esz)) || (e = cudaMalloc(&c.act, B * c.F * c.esz)) ||
      (e = cudaMalloc(&c.attn_out, B * c.qd * c.esz)) || (e = dalloc(&c.qkv, B * c.qkvN)) ||
      (e = dalloc(&c.q, B * c.qd)) ||
      (e = dalloc(&c.attn_m, B * c.nq * c.attn_max_chunks)) ||
      (e = dalloc(&c.attn_l, B * c.nq * c.attn_max_chunks)) ||
      (e = dalloc(&c.attn_acc, B * c.nq * c.attn_max_chunks * c.hd)) ||
      (e = dalloc(&c.attn_ctr, B * c.nkv)) ||
      (e = dalloc(&c.dm_u, (size_t)kRouteZSlots * B * c.r)) || (e = dalloc(&c.dm_x, B * 2 * c.d)) ||
      (e = dalloc(&c.mask, B * c.L)) ||
      (e = dalloc(&c.sel, B * c.Lm)) || (e = dalloc(&c.scores, B * c.Lm)) ||
      (e = dalloc(&c.rows, (size_t)c.L * B)) || (e = dalloc(&c.count, (size_t)c.L)) ||
      (e = dalloc(&c.h_in_stage, B * c.d)) || (e = dalloc(&c.h_out_stage, B * c.d)) ||
      (e = dalloc(&c.k_stage, B)) || (e = dalloc(&c.mask_stage, B * c.L)))
    return fail(e);
  c.split0 = c.dtype == BUDDY_DTYPE_BF16;
  if (c.split0 && ((e = cudaMalloc(&c.xn_lo, B * c.d * c.esz)) || (e = cudaMalloc(&c.act_lo, B * c.F * c.esz)) ||
                   (e = cudaMalloc(&c.attn_lo, B * c.qd * c.esz))))
    return fail(e);
  if ((e = cudaMemset(c.status, 0, 4 * sizeof(int32_t))) != cudaSuccess ||
      (e = cudaMemset(c.attn_ctr, 0, B * c.nkv * sizeof(int32_t))) != cudaSuccess)
    return fail(e);
  c.dm_u_cols = c.r;
  c.pf_max = g.max_prefill_tokens;
  if (c.pf_max > 0) {
    const size_t T = c.pf_max;
    c.pf_items_max = (int64_t)(T / 64 + B) * c.nq;
    if ((e = cudaMalloc(&c.pf_xn, T * c.d * c.esz)) || (e = cudaMalloc(&c.pf_xn_lo, T * c.d * c.esz)) ||
        (e = dalloc(&c.pf_q, T * c.qd)) || (e = cudaMalloc(&c.pf_attn, T * c.qd * c.esz)) ||
        (e = cudaMalloc(&c.pf_attn_lo, T * c.qd * c.esz)) || (e = cudaMalloc(&c.pf_act, T * c.F * c.esz)) ||
        (e = cudaMalloc(&c.pf_act_lo, T * c.F * c.esz)) || (e = dalloc(&c.pf_tok_seq, T)) ||
        (e = dalloc(&c.pf_tok_t, T)) || (e = dalloc(&c.pf_tok_pos, T)) ||
        (e = dalloc(&c.pf_rows, (size_t)c.L * T)) ||
        (e = dalloc(&c.pf_items, (size_t)(c.L + 1) * c.pf_items_max)) || (e = dalloc(&c.pf_n_tok, B)) ||
        (e = dalloc(&c.pf_tok_end, B)) || (e = dalloc(&c.pf_cnt, B)) || (e = dalloc(&c.pf_hlast, B * c.d)))
      return fail(e);
  }
  if ((e = cudaStreamCreateWithFlags(&x->cap_stream, cudaStreamNonBlocking)) != cudaSuccess) return fail(e);
  launch_rope_table(c.rope_cos, c.rope_sin, c.max_pos, c.hd, (double)g.rope_theta, x->cap_stream);
  if ((e = cudaGetLastError()) != cudaSuccess || (e = cudaStreamSynchronize(x->cap_stream)) != cudaSuccess)
    return fail(e);
  *out = x;
  return BUDDY_OK;
}

extern "C" void buddy_destroy(buddy_ctx* ctx) {
  if (!ctx) return;
  cudaDeviceSynchronize();
  free_ctx(ctx);
}

// Device buffers the kernels read or write with 16-byte vector accesses.
static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

extern "C" int buddy_set_weights(buddy_ctx* ctx, const buddy_layer_weights* layers,
                                 const buddy_dm_weights* dm) {
  if (!ctx || !layers || !dm) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  for (int l = 0; l < c.L; ++l) {
    const buddy_layer_weights& w = layers[l];
    if (!w.attn_norm || !w.w_qkv || !w.w_o || !w.ffn_norm || !w.w_gate_up || !w.w_down)
      return BUDDY_ERR_ARG;
    const void* wp[] = {w.attn_norm, w.w_qkv, w.w_o, w.ffn_norm, w.w_gate_up, w.w_down};
    for (const void* p : wp)
      if (!aligned16(p)) return BUDDY_ERR_ARG;
    if (c.cfg.qkv_bias && !w.b_qkv) return BUDDY_ERR_ARG;
  }
  if (!dm->w1 || !dm->b1 || !dm->w2 || !dm->b2) return BUDDY_ERR_ARG;
  c.layers.assign(layers, layers + c.L);
  if (!c.cfg.qkv_bias)
    for (auto& w : c.layers) w.b_qkv = nullptr;
  c.dm = *dm;
  for (auto& kv : c.graphs) cudaGraphExecDestroy(kv.second);
  c.graphs.clear();
  c.have_weights = true;
  const int rc = gemm_tc_prepare(c);
  if (rc != BUDDY_OK) {
    c.have_weights = false;
    return rc;
  }
  return BUDDY_OK;
}

extern "C" int buddy_set_budget_predictor(buddy_ctx* ctx, const buddy_predictor_weights* bp) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (bp && (!bp->w1 || !bp->b1 || !bp->w2 || !bp->b2 || bp->hidden < 1 || bp->hidden > 65536))
    return BUDDY_ERR_ARG;
  CK(cudaDeviceSynchronize());   // dm_u may be in use by queued work
  for (auto& kv : c.graphs) cudaGraphExecDestroy(kv.second);
  c.graphs.clear();
  const int cols = c.r + (bp ? bp->hidden : 0);
  if (cols > c.dm_u_cols) {
    float* nu = nullptr;
    CK(cudaMalloc(&nu, (size_t)kRouteZSlots * c.maxB * cols * sizeof(float)));
    cudaFree(c.dm_u);
    c.dm_u = nu;
    c.dm_u_cols = cols;
  }
  c.have_pred = bp != nullptr;
  if (bp) c.pred = *bp;
  return BUDDY_OK;
}

extern "C" int buddy_set_wait_limit(buddy_ctx* ctx, int64_t ns) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  CK(cudaDeviceSynchronize());
  c.wait_ns = ns > 0 ? (uint64_t)ns : 4000000000ull;
  for (auto& kv : c.graphs) cudaGraphExecDestroy(kv.second);   // the limit is baked into captured launches
  c.graphs.clear();
  return BUDDY_OK;
}

extern "C" int buddy_set_options(buddy_ctx* ctx, int32_t use_graph) {
  if (!ctx) return BUDDY_ERR_ARG;
  ctx->c.use_graph = use_graph ? 1 : 0;
  return BUDDY_OK;
}

static int check_kv(const Ctx& c, const buddy_kv_state* kv, int need_batch) {
  if (!kv || !kv->k_cache || !kv->v_cache || !kv->seq_off || !kv->cap || !kv->len || !kv->pool_sum)
    return BUDDY_ERR_ARG;
  if (c.masked && !kv->layer_len) return BUDDY_ERR_ARG;
  if (kv->batch < need_batch || kv->batch < 1) return BUDDY_ERR_ARG;
  if (!aligned16(kv->pool_sum)) return BUDDY_ERR_ARG;
  for (int l = 0; l < c.L; ++l)
    if (!kv->k_cache[l] || !kv->v_cache[l] || !aligned16(kv->k_cache[l]) || !aligned16(kv->v_cache[l]))
      return BUDDY_ERR_ARG;
  return BUDDY_OK;
}

extern "C" int buddy_device_status(buddy_ctx* ctx, void* stream, int32_t* flags) {
  if (!ctx || !flags) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  cudaStream_t s = (cudaStream_t)stream;
  int32_t h[2] = {0, 0};
  CK(cudaMemcpyAsync(h, c.status, 2 * sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  CK(cudaMemsetAsync(c.status, 0, 2 * sizeof(int32_t), s));
  if (h[0] & BUDDY_DEV_TIMEOUT) {
    // a GEMM that gave up left split-K arrival counters mid-count: re-arm them
    if (c.gemm_ctr) CK(cudaMemsetAsync(c.gemm_ctr, 0, c.gemm_ctr_n * sizeof(int32_t), s));
    CK(cudaMemsetAsync(c.attn_ctr, 0, (size_t)c.maxB * c.nkv * sizeof(int32_t), s));
  }
  CK(cudaStreamSynchronize(s));
  *flags = h[0];
  return h[0] ? BUDDY_ERR_DEVICE : BUDDY_OK;
}

extern "C" int buddy_get_paths(buddy_ctx* ctx, int32_t* paths, int32_t n) {
  if (!ctx || !paths || n < 0 || n > 4) return BUDDY_ERR_ARG;
  const Ctx& c = ctx->c;
  if (!c.have_weights) return BUDDY_ERR_STATE;
  const int32_t v[4] = {c.use_tc ? 1 : 0, attention_cl(c) ? 2 : (attention_tc(c) ? 1 : 0),
                        (c.use_tc && c.tc_panel) ? 1 : 0,
                        (c.use_tc && c.tc_defer) ? 1 : 0};
  for (int i = 0; i < n; ++i) paths[i] = v[i];
  return BUDDY_OK;
}

extern "C" int buddy_set_profiling(buddy_ctx* ctx, int32_t on) {
  if (!ctx) return BUDDY_ERR_ARG;
  ctx->c.profiling = on ? 1 : 0;
  return BUDDY_OK;
}

extern "C" const char* buddy_profile_class_name(int32_t cls) {
  static const char* names[BUDDY_PROF_NCLASS] = {"check", "rmsnorm", "gemm_qkv", "qkv_finalize",
                                                 "attention", "gemm_o", "gemm_gate_up", "gemm_down",
                                                 "route", "compact", "other", "gemm_fixup",
                                                 "pf_gemm", "pf_attention", "pf_other"};
  return (cls >= 0 && cls < BUDDY_PROF_NCLASS) ? names[cls] : "unknown";
}

extern "C" int buddy_profile_read(buddy_ctx* ctx, int32_t n_cls, float* ms, int32_t* launches) {
  if (!ctx || n_cls < 0 || n_cls > BUDDY_PROF_NCLASS || (n_cls > 0 && (!ms || !launches)))
    return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  for (int i = 0; i < n_cls; ++i) {
    ms[i] = 0.f;
    launches[i] = 0;
  }
  for (const auto& r : c.prof) {
    CK(cudaEventSynchronize(r.b));
    float t = 0.f;
    CK(cudaEventElapsedTime(&t, r.a, r.b));
    if (r.cls < n_cls) {
      ms[r.cls] += t;
      launches[r.cls] += r.launches;
    }
  }
  c.prof.clear();
  c.ev_used = 0;
  return BUDDY_OK;
}

// ---------------------------------------------------------------------------
// GEMM dispatch
// ---------------------------------------------------------------------------
static void run_gemm(Ctx& c, int epi, GemmArgs a, int layer, int which, cudaStream_t s, int cls, bool prof) {
  a.status = c.status;
  a.layer = layer;
  a.which = which;
  if (c.use_tc) {
    {
      ProfScope p(c, s, cls, 1, prof);
      launch_gemm_tc(c, epi, a, s);
    }
    // (a SwiGLU GEMM with one K split applies its epilogue itself)
    if (c.tc_defer && !(epi == EPI_SWIGLU && c.tc_splits[which] == 1)) {
      ProfScope p(c, s, BUDDY_PROF_GEMM_FIXUP, 1, prof);
      launch_gemm_fix(c, epi, a, s);
    }
  } else {
    ProfScope p(c, s, cls, 1, prof);
    launch_gemm_simt(c, epi, a, s);
  }
}

// GEMM arguments of one decoder block (Eq. 1 executed branch) on the rows of
// `sel`: the residual stream H is updated in place for those rows; `src` is
// the block's input (h_in for layer 0, else H).  Layers 0..c feed the router:
// their GEMM inputs are kept as bf16 hi + lo pairs (split) so that the
// routing input carries ~16 mantissa bits.  With `panel` the RMSNorms run
// inside the QKV and gate/up GEMMs.
static GemmArgs qkv_args(const Ctx& c, const buddy_kv_state& kv, int l, RowSel sel, const float* src, bool split,
                         bool panel) {
  const buddy_layer_weights& W = c.layers[l];
  GemmArgs g{};
  g.sel = sel;
  g.max_m = sel.n;
  g.split = split;
  g.W = W.w_qkv; g.X = c.xn; g.X_lo = c.xn_lo; g.N = c.qkvN; g.K = c.d; g.out_f32 = c.qkv;
  if (panel) {
    g.in_norm_src = src;
    g.in_norm_gamma = W.attn_norm;
  }
  // the value-state feature is pooled with the QKV finalisation of the
  // context layer, the other features by launch_pool_update
  g.pool = (l == c.cl && c.feature == BUDDY_FEATURE_V) ? kv.pool_sum : nullptr;
  if (c.use_tc) {
    // bias, RoPE, q, cache append and pool update in the GEMM epilogue
    g.qkv_bias = W.b_qkv; g.kv_len = kv.len; g.kv_seq_off = kv.seq_off; g.kv_cap = kv.cap;
    g.cache_len = cache_len(c, kv, l);
    g.kc = kv.k_cache[l]; g.vc = kv.v_cache[l]; g.q_out = c.q;
  }
  g.status = c.status;
  g.layer = l;
  g.which = 0;
  return g;
}
static GemmArgs o_args(const Ctx& c, int l, RowSel sel, const float* src, float* H, bool split) {
  GemmArgs g{};
  g.sel = sel; g.max_m = sel.n; g.split = split;
  g.W = c.layers[l].w_o; g.X = c.attn_out; g.X_lo = c.attn_lo; g.N = c.d; g.K = c.qd;
  g.resid_src = src; g.resid_dst = H;
  g.status = c.status; g.layer = l; g.which = 1;
  return g;
}
static GemmArgs gate_up_args(const Ctx& c, int l, RowSel sel, float* H, bool split, bool panel) {
  GemmArgs g{};
  g.sel = sel; g.max_m = sel.n; g.split = split;
  g.W = c.layers[l].w_gate_up; g.X = c.xn; g.X_lo = c.xn_lo; g.N = c.F; g.K = c.d; g.out_act = c.act;
  if (panel) {
    g.in_norm_src = H;
    g.in_norm_gamma = c.layers[l].ffn_norm;
  }
  g.out_act_lo = split ? c.act_lo : nullptr;
  g.status = c.status; g.layer = l; g.which = 2;
  return g;
}
static GemmArgs down_args(const Ctx& c, int l, RowSel sel, float* H, bool split) {
  GemmArgs g{};
  g.sel = sel; g.max_m = sel.n; g.split = split;
  g.W = c.layers[l].w_down; g.X = c.act; g.X_lo = c.act_lo; g.N = c.d; g.K = c.F;
  g.resid_src = H; g.resid_dst = H;
  g.status = c.status; g.layer = l; g.which = 3;
  return g;
}

static void enqueue_attention(Ctx& c, const buddy_kv_state& kv, int l, RowSel sel, bool split, cudaStream_t s,
                              bool prof) {
  ProfScope p(c, s, BUDDY_PROF_ATTENTION, 1, prof);
  launch_attention(c, sel, kv, l, c.q, c.attn_out, split ? c.attn_lo : nullptr, s);
}

// One decoder block, one launch per GEMM.
static void enqueue_layer(Ctx& c, const buddy_kv_state& kv, int l, RowSel sel, const float* src,
                          float* H, cudaStream_t s, bool prof) {
  const buddy_layer_weights& W = c.layers[l];
  const bool split = c.split0 && l <= c.cl;
  const bool panel = c.use_tc && c.tc_panel;
  if (!panel) {
    ProfScope p(c, s, BUDDY_PROF_RMSNORM, 1, prof);
    launch_rmsnorm(c, src, sel, W.attn_norm, c.xn, split ? c.xn_lo : nullptr, s);
  }
  GemmArgs g = qkv_args(c, kv, l, sel, src, split, panel);
  // no RMSNorm kernel in between: the first middle layer's QKV GEMM follows
  // the compaction kernel that writes its row count
  g.count_late = panel && l == c.cl + 1;
  if (c.use_tc) {
    run_gemm(c, EPI_QKV, g, l, 0, s, BUDDY_PROF_GEMM_QKV, prof);
  } else {
    run_gemm(c, EPI_STORE_F32, g, l, 0, s, BUDDY_PROF_GEMM_QKV, prof);
    ProfScope p(c, s, BUDDY_PROF_QKV_FINALIZE, 1, prof);
    launch_qkv_finalize(c, c.qkv, W.b_qkv, sel, kv, l, c.q, g.pool, s);
  }
  enqueue_attention(c, kv, l, sel, split, s, prof);
  run_gemm(c, EPI_RESID, o_args(c, l, sel, src, H, split), l, 1, s, BUDDY_PROF_GEMM_O, prof);
  if (!panel) {
    ProfScope p(c, s, BUDDY_PROF_RMSNORM, 1, prof);
    launch_rmsnorm(c, H, sel, W.ffn_norm, c.xn, split ? c.xn_lo : nullptr, s);
  }
  run_gemm(c, EPI_SWIGLU, gate_up_args(c, l, sel, H, split, panel), l, 2, s, BUDDY_PROF_GEMM_GATE_UP, prof);
  run_gemm(c, EPI_RESID, down_args(c, l, sel, H, split), l, 3, s, BUDDY_PROF_GEMM_DOWN, prof);
}

struct StepIO {
  int B;
  const float* h_in;
  const int32_t* k;
  float* h_out;
  uint8_t* mask_out;
  int32_t* rows_out;
  int32_t* count_out;
  float* scores_out;
};

// Enqueues the whole step on `s` (which the caller may be capturing into a
// graph).  With profiling, the host reads the layer counts and launches only
// the layers some sequence selected.
static int enqueue_step(buddy_ctx* x, const buddy_kv_state& kv, const StepIO& io, cudaStream_t s,
                        bool capture) {
  Ctx& c = x->c;
  const int B = io.B;
  const bool prof = c.profiling && !capture;
  {
    ProfScope p(c, s, BUDDY_PROF_CHECK, 1, prof);
    launch_step_check(c, B, io.k, kv, 1, c.status, s);
  }
  const RowSel all{nullptr, nullptr, B};
  for (int l = 0; l <= c.cl; ++l) enqueue_layer(c, kv, l, all, l == 0 ? io.h_in : io.h_out, io.h_out, s, prof);
  if (c.feature != BUDDY_FEATURE_V) {
    ProfScope p(c, s, BUDDY_PROF_ROUTE, 1, prof);
    launch_pool_update(c, B, kv, s);
  }
  {
    ProfScope p(c, s, BUDDY_PROF_ROUTE, 2, prof);
    launch_route(c, B, io.h_out, kv.pool_sum, kv.len, 1, io.k, c.mask, c.sel, c.scores, s);
  }
  {
    ProfScope p(c, s, BUDDY_PROF_COMPACT, 1, prof);
    launch_compact(c, B, c.mask, kv, c.rows, c.count, s);
  }
  int32_t hcount[kMaxLayers];
  if (prof) {
    // profiling: launch only the layers some sequence selected
    CK(cudaMemcpyAsync(hcount, c.count, sizeof(int32_t) * c.L, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
  }
  // Every middle layer is enqueued; a layer that no sequence selected costs one
  // early exit per kernel (its row count, written by the compaction kernel, is
  // read before any setup).  Graph conditional nodes would skip those launches
  // but cut the programmatic-dependent-launch overlap at every executed layer,
  // which costs more at the budgets of interest.
  for (int l = c.cl + 1; l < c.L - 1; ++l) {
    const RowSel sel{c.rows + (size_t)l * B, c.count + l, B};
    if (!prof || hcount[l] > 0) enqueue_layer(c, kv, l, sel, io.h_out, io.h_out, s, prof);
  }
  enqueue_layer(c, kv, c.L - 1, all, io.h_out, io.h_out, s, prof);
  {
    ProfScope p(c, s, BUDDY_PROF_OTHER, 1, prof);
    launch_advance(c, B, kv.len, 1, nullptr, s, c.masked ? c.mask : nullptr, kv.layer_len, kv.batch);
  }
  if (io.mask_out) CK(cudaMemcpyAsync(io.mask_out, c.mask, (size_t)B * c.L, cudaMemcpyDeviceToDevice, s));
  if (io.rows_out)
    CK(cudaMemcpyAsync(io.rows_out, c.rows, (size_t)B * c.L * sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
  if (io.count_out)
    CK(cudaMemcpyAsync(io.count_out, c.count, (size_t)c.L * sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
  if (io.scores_out)
    CK(cudaMemcpyAsync(io.scores_out, c.scores, (size_t)B * c.Lm * sizeof(float), cudaMemcpyDeviceToDevice, s));
  CK(cudaGetLastError());
  return BUDDY_OK;
}

static int run_step(buddy_ctx* x, const buddy_kv_state* kv, const StepIO& io, cudaStream_t s) {
  Ctx& c = x->c;
  if (!c.use_graph) return enqueue_step(x, *kv, io, s, false);
  Ctx::GraphKey key{io.B, io.h_in, io.k, io.h_out, io.mask_out, io.rows_out, io.count_out,
                    io.scores_out, s, {}};
  for (int l = 0; l < c.L; ++l) {
    key.kvp.push_back(kv->k_cache[l]);
    key.kvp.push_back(kv->v_cache[l]);
  }
  key.kvp.push_back(kv->seq_off);
  key.kvp.push_back(kv->cap);
  key.kvp.push_back(kv->len);
  key.kvp.push_back(kv->pool_sum);
  key.kvp.push_back(kv->layer_len);
  auto it = c.graphs.find(key);
  if (it == c.graphs.end()) {
    if (c.graphs.size() >= 16) {   // bounded cache: drop an arbitrary old entry
      CK(cudaStreamSynchronize(s));
      cudaGraphExecDestroy(c.graphs.begin()->second);
      c.graphs.erase(c.graphs.begin());
    }
    cudaStream_t cs = x->cap_stream;
    CK(cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed));
    int rc = enqueue_step(x, *kv, io, cs, true);
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamEndCapture(cs, &g);
    if (rc != BUDDY_OK) {
      if (g) cudaGraphDestroy(g);
      return rc;
    }
    CK(e);
    cudaGraphExec_t ge = nullptr;
    e = cudaGraphInstantiate(&ge, g, 0);
    cudaGraphDestroy(g);
    CK(e);
    it = c.graphs.emplace(key, ge).first;
  }
  CK(cudaGraphLaunch(it->second, s));
  return BUDDY_OK;
}

extern "C" int buddy_decode_step(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch,
                                 const float* h_in, const int32_t* k, float* h_out,
                                 uint8_t* mask_out, int32_t* rows_out, int32_t* count_out,
                                 float* scores_out, void* stream) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (!c.have_weights) return BUDDY_ERR_STATE;
  if (batch < 1 || batch > c.maxB || !h_in || !k || !h_out || h_in == h_out) return BUDDY_ERR_ARG;
  if (!aligned16(h_in) || !aligned16(h_out)) return BUDDY_ERR_ARG;
  int rc = check_kv(c, kv, batch);
  if (rc) return rc;
  StepIO io{batch, h_in, k, h_out, mask_out, rows_out, count_out, scores_out};
  return run_step(ctx, kv, io, (cudaStream_t)stream);
}

extern "C" int buddy_decode_step_host(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch,
                                      const float* h_in_host, const int32_t* k_host,
                                      float* h_out_host, uint8_t* mask_host, void* stream) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (!c.have_weights) return BUDDY_ERR_STATE;
  if (batch < 1 || batch > c.maxB || !h_in_host || !k_host || !h_out_host) return BUDDY_ERR_ARG;
  int rc = check_kv(c, kv, batch);
  if (rc) return rc;
  cudaStream_t s = (cudaStream_t)stream;
  CK(cudaMemcpyAsync(c.h_in_stage, h_in_host, (size_t)batch * c.d * sizeof(float), cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(c.k_stage, k_host, (size_t)batch * sizeof(int32_t), cudaMemcpyHostToDevice, s));
  StepIO io{batch, c.h_in_stage, c.k_stage, c.h_out_stage, mask_host ? c.mask_stage : nullptr,
            nullptr, nullptr, nullptr};
  rc = run_step(ctx, kv, io, s);
  if (rc) return rc;
  CK(cudaMemcpyAsync(h_out_host, c.h_out_stage, (size_t)batch * c.d * sizeof(float), cudaMemcpyDeviceToHost, s));
  if (mask_host) CK(cudaMemcpyAsync(mask_host, c.mask_stage, (size_t)batch * c.L, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  return BUDDY_OK;
}

extern "C" int buddy_prefill(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch, const int32_t* n_tok,
                             const float* x, const int32_t* k, float* h_out, uint8_t* mask_out, float* scores_out,
                             void* stream) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (!c.have_weights) return BUDDY_ERR_STATE;
  if (c.pf_max <= 0 || c.dtype != BUDDY_DTYPE_BF16) return BUDDY_ERR_STATE;
  if (batch < 1 || batch > c.maxB || !n_tok || !x || !k || !h_out || x == h_out) return BUDDY_ERR_ARG;
  if (!aligned16(x) || !aligned16(h_out)) return BUDDY_ERR_ARG;
  int rc = check_kv(c, kv, batch);
  if (rc) return rc;
  int64_t T = 0;
  for (int i = 0; i < batch; ++i) {
    if (n_tok[i] < 1) return BUDDY_ERR_RANGE;
    T += n_tok[i];
  }
  if (T > c.pf_max) return BUDDY_ERR_RANGE;
  return run_prefill(c, *kv, batch, n_tok, x, k, h_out, mask_out, scores_out, (cudaStream_t)stream);
}

extern "C" int buddy_route(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t batch, const float* h1,
                           const int32_t* k, int32_t* sel_out, uint8_t* mask_out, float* scores_out,
                           void* stream) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (!c.have_weights) return BUDDY_ERR_STATE;
  if (batch < 1 || batch > c.maxB || !h1 || !k || !aligned16(h1)) return BUDDY_ERR_ARG;
  if (!kv || !kv->len || !kv->pool_sum || !kv->cap || kv->batch < batch) return BUDDY_ERR_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  // positions: the cache already holds the newest token (len >= 1)
  buddy_kv_state kvc = *kv;
  kvc.layer_len = nullptr;   // only the context layer's pool and len are read
  launch_step_check(c, batch, k, kvc, 0, c.status, s);
  launch_route(c, batch, h1, kv->pool_sum, kv->len, 0, k, mask_out, sel_out, scores_out, s);
  CK(cudaGetLastError());
  return BUDDY_OK;
}

extern "C" int buddy_kv_append(buddy_ctx* ctx, const buddy_kv_state* kv, int32_t layer,
                               int32_t n_seq, const int32_t* seq_ids, int32_t n_new,
                               const void* k_new, const void* v_new, int32_t advance, void* stream) {
  if (!ctx) return BUDDY_ERR_ARG;
  Ctx& c = ctx->c;
  if (layer < 0 || layer >= c.L || n_seq < 1 || n_seq > kMaxBatch * 64 || n_new < 0 || !seq_ids)
    return BUDDY_ERR_ARG;
  if (n_new > 0 && (!k_new || !v_new)) return BUDDY_ERR_ARG;
  if (n_new > 65535) return BUDDY_ERR_RANGE;
  int rc = check_kv(c, kv, 1);
  if (rc) return rc;
  cudaStream_t s = (cudaStream_t)stream;
  int32_t* base = const_cast<int32_t*>(cache_len(c, *kv, layer));
  launch_kv_check(c, n_seq, seq_ids, n_new, kv->batch, base, kv->cap, c.status, s);
  if (n_new > 0) launch_kv_append(c, *kv, layer, n_seq, seq_ids, n_new, k_new, v_new, s);
  if (layer == c.cl) launch_pool_refresh(c, *kv, n_seq, seq_ids, n_new, s);
  // the masked variant's per-layer length grows with its own appends
  if (c.masked && n_new > 0) launch_advance(c, n_seq, base, n_new, seq_ids, s);
  if (advance && n_new > 0) launch_advance(c, n_seq, kv->len, n_new, seq_ids, s);
  CK(cudaGetLastError());
  return BUDDY_OK;
}

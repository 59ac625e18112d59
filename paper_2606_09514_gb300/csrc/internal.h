// Host-side internals of libbuddy: context layout and kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <map>
#include <utility>
#include <vector>

#include "../../include/buddy.h"

namespace buddy {

constexpr int kMaxLayers = 128;
constexpr int kRouteZSlots = 16;  // K-split slots of the router's hidden-unit partial sums
constexpr int kMaxBatch = 1024;

// Per-layer K/V base pointers passed by value to kernels that touch many layers.
struct LayerPtrs {
  void* k[kMaxLayers];
  void* v[kMaxLayers];
};

// Where the row list of a layer comes from: identity (rows == nullptr) with a
// fixed count, or a device list with a device count.
struct RowSel {
  const int32_t* rows;    // device [max_batch] or nullptr (identity)
  const int32_t* count;   // device scalar or nullptr (use n)
  int n;                  // count when `count` is null; upper bound otherwise
};

enum GemmEpi { EPI_STORE_F32 = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };

struct GemmArgs {
  const void* W;          // [N_rows, K] (weight dtype)
  const void* X;          // [m, K] compact activations (act dtype)
  int N;                  // output features (for SWIGLU: F, with W of 2F rows)
  int K;
  RowSel sel;             // m = row count; rows map j -> sequence for EPI_RESID
  int max_m;              // grid sizing bound
  // epilogues
  float* out_f32;         // EPI_STORE_F32: [m, N]
  void* out_act;          // EPI_SWIGLU: [m, N] act dtype
  void* X_lo;             // split activations: bf16 remainder of X (or null)
  void* out_act_lo;       // split activations: bf16 remainder of the SwiGLU output
  bool split;
  const float* resid_src; // EPI_RESID: dst[i] = src[i] + acc  (may equal dst)
  float* resid_dst;
  // EPI_QKV (tensor-core path): QKV finalisation fused into the epilogue
  const float* qkv_bias;
  const int32_t* kv_len;       // RoPE positions (tokens of each sequence)
  const int32_t* cache_len;    // where the layer's cache stores the new entry
  const int64_t* kv_seq_off;
  const int32_t* kv_cap;
  void* kc;
  void* vc;
  float* q_out;
  float* pool;
  const int32_t* status;
  int layer;              // tensor-core path: which layer's weight map
  int which;              // 0 qkv, 1 o, 2 gate_up, 3 down
  // tensor-core path, small batches: X = RMSNorm(in_norm_src[rows]) computed
  // inside the GEMM (panel mode; X and X_lo unused)
  const float* in_norm_src;
  const float* in_norm_gamma;
  bool count_late;        // the kernel enqueued just before wrote *sel.count
};

struct Ctx;

// Epilogue pointers of a prefill GEMM (gemm_pf.cu); unused ones stay null.
struct PfEpi {
  const int32_t* rows;      // compact row -> token row (nullptr: identity)
  const float* resid_src;
  float* resid_dst;
  void* out_act;
  void* out_act_lo;
  float* q_out;
  const float* bias;
  const int32_t* tok_seq;
  const int32_t* tok_pos;
  const int32_t* len;
  const int32_t* cache_len;
  const int64_t* seq_off;
  const int32_t* cap;
  void* kc;
  void* vc;
};

// Launch with programmatic stream serialisation when `pdl` is set (the kernel
// then overlaps its prologue with the predecessor and synchronises with
// pdl_wait()).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                            bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = pdl ? attr : nullptr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// Kernel launchers (kernels.cu)
void launch_rope_table(float* cos_t, float* sin_t, int max_pos, int hd, double theta, cudaStream_t s);
void launch_step_check(const Ctx& c, int B, const int32_t* k, const buddy_kv_state& kv, int extra_pos,
                       int32_t* status, cudaStream_t s);
void launch_kv_check(const Ctx& c, int n_seq, const int32_t* seq_ids, int n_new, int batch,
                     const int32_t* len, const int32_t* cap, int32_t* status, cudaStream_t s);
void launch_rmsnorm(const Ctx& c, const float* H, RowSel sel, const float* gamma, void* xn, void* xn_lo,
                    cudaStream_t s);
void launch_qkv_finalize(const Ctx& c, const float* qkv, const float* bias, RowSel sel,
                         const buddy_kv_state& kv, int layer, float* q_out, float* pool,
                         cudaStream_t s);
void launch_attention(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q,
                      void* attn_out, void* attn_lo, cudaStream_t s);   // attention.cu
int attention_max_spans(int max_pos);   // span partials per (row, query head)
bool attention_tc(const Ctx& c);         // tensor-core loop over the whole GPU
bool attention_cl(const Ctx& c);         // small batches: one cluster per stream (attn_cl.cu)
void launch_attention_cl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q, void* out,
                         void* out_lo, cudaStream_t s);
void launch_route(const Ctx& c, int B, const float* h1, const float* pool, const int32_t* len,
                  int len_bias, const int32_t* k, uint8_t* mask, int32_t* sel, float* scores,
                  cudaStream_t s);
void launch_compact(const Ctx& c, int B, const uint8_t* mask, const buddy_kv_state& kv,
                    int32_t* rows, int32_t* count, cudaStream_t s);
void launch_advance(const Ctx& c, int B, int32_t* len, int by, const int32_t* seq_ids, cudaStream_t s,
                    const uint8_t* mask = nullptr, int32_t* layer_len = nullptr, int kv_batch = 0);
void launch_pool_update(const Ctx& c, int B, const buddy_kv_state& kv, cudaStream_t s);
void launch_kv_append(const Ctx& c, const buddy_kv_state& kv, int layer, int n_seq,
                      const int32_t* seq_ids, int n_new, const void* k_new, const void* v_new,
                      cudaStream_t s);
void launch_pool_refresh(const Ctx& c, const buddy_kv_state& kv, int n_seq, const int32_t* seq_ids,
                         int n_new, cudaStream_t s);
// GEMMs (gemm_simt.cu, gemm_tc.cu)
void launch_gemm_simt(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s);
bool gemm_tc_supported(const Ctx& c);
void launch_gemm_tc(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s);
// prefill (gemm_pf.cu, attn_pf.cu, prefill.cu)
int gemm_pf_prepare(Ctx& c);
void launch_gemm_pf(const Ctx& c, int epi, bool split, int layer, int which, int xi, int m, const PfEpi& e,
                    cudaStream_t s);
void launch_attention_pf(const Ctx& c, int n_items, const int4* items, const int32_t* n_tok, const int32_t* base,
                         const buddy_kv_state& kv, int layer, const float* q, void* out, void* out_lo,
                         cudaStream_t s);
void launch_pool_refresh_n(const Ctx& c, const buddy_kv_state& kv, int n_seq, const int32_t* n_new,
                           cudaStream_t s);
int run_prefill(Ctx& c, const buddy_kv_state& kv, int B, const int32_t* n_tok_host, const float* x,
                const int32_t* k, float* h_out, uint8_t* mask_out, float* scores_out, cudaStream_t s);
void launch_gemm_fix(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s);   // with c.tc_defer

struct Ctx {
  buddy_config cfg;
  // Lm = n_cand, the routed layers cl+1 .. L-2 (cl = the context layer)
  int L, Lm, cl, d, nq, nkv, hd, F, r, qd, kvd, qkvN, maxB, max_pos;
  int dtype;
  int feature = BUDDY_FEATURE_V;   // planner feature
  bool masked = false;             // BUDDY_SKIP_MASKED: per-layer cache lengths
  size_t esz;
  int device, num_sms;
  bool pdl = true;             // programmatic dependent launch between step kernels
  uint64_t wait_ns = 4000000000ull;   // limit of each bounded wait in the GEMM pipelines

  bool have_weights = false;
  std::vector<buddy_layer_weights> layers;
  buddy_dm_weights dm{};
  bool have_pred = false;          // Budget Predictor registered
  buddy_predictor_weights pred{};
  int dm_u_cols = 0;               // columns of dm_u: r + predictor hidden

  // scratch (device)
  float* rope_cos = nullptr;   // [max_pos, hd/2]
  float* rope_sin = nullptr;
  int32_t* status = nullptr;   // [0] sticky bits, [1] abort flag, [2..] spare
  void* xn = nullptr;          // [maxB, d]   act dtype: normalised GEMM input
  void* act = nullptr;         // [maxB, F]   act dtype: SwiGLU output
  void* attn_out = nullptr;    // [maxB, qd]  act dtype
  // first layer (the router's input) keeps activations as bf16 hi + lo pairs
  bool split0 = false;
  void* xn_lo = nullptr;       // [maxB, d]
  void* act_lo = nullptr;      // [maxB, F]
  void* attn_lo = nullptr;     // [maxB, qd]
  float* qkv = nullptr;        // [maxB, qkvN]
  float* q = nullptr;          // [maxB, qd]
  int attn_max_chunks = 1;   // span partial slots per (row, query head)
  float* attn_m = nullptr;     // [maxB, nq, max_chunks]
  float* attn_l = nullptr;
  float* attn_acc = nullptr;   // [maxB, nq, max_chunks, hd]
  int32_t* attn_ctr = nullptr; // [maxB, nkv] chunk arrivals (self-resetting)
  float* dm_u = nullptr;       // [kRouteZSlots, maxB, r + predictor hidden] partial sums
  float* dm_x = nullptr;       // [maxB, 2d] router inputs (larger batches)
  uint8_t* mask = nullptr;     // [maxB, L]
  int32_t* sel = nullptr;      // [maxB, Lm]
  float* scores = nullptr;     // [maxB, Lm]
  int32_t* rows = nullptr;     // [L, maxB]
  int32_t* count = nullptr;    // [L]
  // host-buffer entry staging
  float* h_in_stage = nullptr;
  float* h_out_stage = nullptr;
  int32_t* k_stage = nullptr;
  uint8_t* mask_stage = nullptr;

  // tcgen05 GEMM resources
  bool use_tc = false;
  std::vector<CUtensorMap> tmaps_host;    // per layer 4 weight maps, then 3 activation maps
  int tc_bw = 256, tc_mt = 1, tc_rows_max = 16, tc_acc_bufs = 2;   // tile geometry (gemm_common.cuh)
  int tc_stages[2] = {1, 1}, tc_smem[2] = {0, 0};                   // [plain, split activations]
  uint32_t tc_stage_bytes[2] = {0, 0}, tc_w_off[2] = {0, 0}, tc_xr = 0, tc_tmem_cols = 512;
  int tc_splits[4] = {1, 1, 1, 1}, tc_tiles[4] = {1, 1, 1, 1};
  float* gemm_ws = nullptr;
  size_t gemm_ws_elems = 0;
  int32_t* gemm_ctr = nullptr;
  int gemm_ctr_n = 0;
  // panel mode: the RMSNorms before the QKV and gate/up GEMMs run inside them
  bool tc_panel = false;
  int tc_panel_kb = 0, tc_pstages[2] = {1, 1}, tc_psmem[2] = {0, 0};
  uint32_t tc_panel_bytes[2] = {0, 0};
  // deferred split-K fixup (batches above kTcDeferRows rows): a second kernel
  // per GEMM sums the partials and applies the epilogue on every SM
  bool tc_defer = false;

  // prefill scratch (max_prefill_tokens rows)
  int pf_max = 0;
  int64_t pf_items_max = 0;       // attention work items per block
  void* pf_xn = nullptr;          // [pf_max, d] bf16, and its remainder term
  void* pf_xn_lo = nullptr;
  float* pf_q = nullptr;          // [pf_max, qd]
  void* pf_attn = nullptr;        // [pf_max, qd] bf16 (+ remainder)
  void* pf_attn_lo = nullptr;
  void* pf_act = nullptr;         // [pf_max, F] bf16 (+ remainder)
  void* pf_act_lo = nullptr;
  int32_t* pf_tok_seq = nullptr;  // [pf_max] token row -> sequence
  int32_t* pf_tok_t = nullptr;    // [pf_max] token row -> index in its prompt
  int32_t* pf_tok_pos = nullptr;  // [pf_max] token row -> position
  int32_t* pf_rows = nullptr;     // [L, pf_max] row lists of the routed blocks
  int4* pf_items = nullptr;       // [(L + 1) * pf_items_max] attention work items
  int32_t* pf_n_tok = nullptr;    // [maxB]
  int32_t* pf_tok_end = nullptr;  // [maxB] one past the last token row of each prompt
  int32_t* pf_cnt = nullptr;      // [maxB] positions the pooled context covers
  float* pf_hlast = nullptr;      // [maxB, d] last prompt token's hidden state
  CUtensorMap pf_tmaps[6];        // pf_xn, pf_attn, pf_act, then their remainder terms
  int pf_stages[2] = {1, 1}, pf_smem[2] = {0, 0};

  // profiler: event pairs around kernel launches (direct-launch mode only)
  int profiling = 0;
  struct ProfRec { int cls; int launches; cudaEvent_t a, b; };
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;

  // graph cache
  int use_graph = 0;
  struct GraphKey {
    int B; const void* h_in; const void* k; void* h_out; void* mask; void* rows; void* count;
    void* scores; cudaStream_t stream; std::vector<const void*> kvp;
    bool operator<(const GraphKey& o) const;
  };
  std::map<GraphKey, cudaGraphExec_t> graphs;
};

// ---------------------------------------------------------------------------
// Profiler: an event pair around each launch group (direct-launch mode only).
// ---------------------------------------------------------------------------
inline cudaEvent_t take_event(Ctx& c) {
  if (c.ev_used == c.ev_pool.size()) {
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    c.ev_pool.push_back(e);
  }
  return c.ev_pool[c.ev_used++];
}

struct ProfScope {
  Ctx& c;
  cudaStream_t s;
  Ctx::ProfRec rec{};
  bool on;
  ProfScope(Ctx& c_, cudaStream_t s_, int cls, int launches, bool on_) : c(c_), s(s_), on(on_) {
    if (!on) return;
    rec.cls = cls;
    rec.launches = launches;
    rec.a = take_event(c);
    rec.b = take_event(c);
    on = rec.a && rec.b;
    if (on) cudaEventRecord(rec.a, s);
  }
  ~ProfScope() {
    if (!on) return;
    cudaEventRecord(rec.b, s);
    c.prof.push_back(rec);
  }
};

// Positions layer l holds for each sequence (where its next entry goes):
// layer_len[l] in the masked variant, else len.
inline const int32_t* cache_len(const Ctx& c, const buddy_kv_state& kv, int l) {
  return c.masked ? kv.layer_len + (size_t)l * kv.batch : kv.len;
}

}  // namespace buddy

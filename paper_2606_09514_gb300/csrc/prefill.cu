// Routed prefill (Sec. 4.1; App. E "Prefill vs. Decode"): a batch of prompts
// passes blocks 0..c token by token with causal attention; each prompt is
// routed once, from its pooled context-layer cache (the prompt included) and
// its last token's hidden state after block c; the routed blocks each run on
// every token of the prompts that selected them (grouping by mask, App. C.1);
// a prompt that skips a block stores zero K/V at all its positions there (or
// nothing, in the masked variant).
//
// The host orchestrates one call: the token tables go to the device, blocks
// 0..c and the router run, then one synchronisation brings the routes back so
// that the host can size every later launch exactly (row lists and attention
// work items per block) instead of launching empty tiles.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace buddy {

// ---------------------------------------------------------------------------
// Token tables, checks, gathers and the position advance
// ---------------------------------------------------------------------------
__global__ void pf_tokens_kernel(int T, const int32_t* tok_seq, const int32_t* tok_t, const int32_t* len,
                                 int32_t* tok_pos, const int32_t* status) {
  if (call_aborted(status)) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r < T) tok_pos[r] = len[tok_seq[r]] + tok_t[r];
}

// Budgets in range (0 allowed with a Budget Predictor), and room for every
// prompt: len + n_tok <= cap and <= max_pos (masked variant: every layer's
// length within [0, len]).  Publishes the call's abort word.
__global__ void pf_check_kernel(int B, const int32_t* k, int Lm, int k_min, const int32_t* n_tok,
                                const int32_t* len, const int32_t* cap, int max_pos, const int32_t* layer_len, int L,
                                int kv_batch, int32_t* status) {
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  int b = 0;
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    const int ki = k[i];
    if (ki < k_min || ki > Lm) b |= BUDDY_DEV_BAD_BUDGET;
    const int n = len[i], t = n_tok[i];
    if (n < 0 || n + t > cap[i] || n + t > max_pos) b |= BUDDY_DEV_BAD_POSITION;
    if (layer_len != nullptr)
      for (int l = 0; l < L; ++l) {
        const int nl = layer_len[(size_t)l * kv_batch + i];
        if (nl < 0 || nl > n) b |= BUDDY_DEV_BAD_POSITION;
      }
  }
  if (b) atomicOr(&bad, b);
  __syncthreads();
  if (threadIdx.x == 0) {
    status[1] = bad ? 1 : 0;
    if (bad) atomicOr(status, bad);
  }
}

// The router's inputs: the last prompt token's hidden state per sequence and
// the number of positions the pooled context covers (len + n_tok).
__global__ void pf_gather_kernel(int B, int d, const int32_t* tok_end, const float* H, const int32_t* len,
                                 const int32_t* n_tok, float* hlast, int32_t* cnt, const int32_t* status) {
  if (call_aborted(status)) return;
  const int i = blockIdx.x;
  const float* src = H + (size_t)(tok_end[i] - 1) * d;
  for (int e = threadIdx.x; e < d; e += blockDim.x) hlast[(size_t)i * d + e] = src[e];
  if (threadIdx.x == 0) cnt[i] = len[i] + n_tok[i];
}

// Zero K and V at every prompt position of the routed blocks a prompt skips.
template <typename T>
__global__ void pf_zero_kernel(int B, int L, int first, int nkv, int hd, const uint8_t* mask, LayerPtrs ptrs,
                               const int32_t* len, const int32_t* n_tok, const int64_t* seq_off,
                               const int32_t* cap, const int32_t* status) {
  if (call_aborted(status)) return;
  const int l = first + blockIdx.x, i = blockIdx.y;
  if (l >= L - 1 || mask[(size_t)i * L + l]) return;
  T* Kc = (T*)ptrs.k[l];
  T* Vc = (T*)ptrs.v[l];
  const int n = n_tok[i], p0 = len[i];
  for (int g = 0; g < nkv; ++g) {
    const int64_t base = kv_offset(seq_off, cap, i, nkv, hd, g, p0);
    for (int x = threadIdx.x; x < n * hd; x += blockDim.x) {
      Kc[base + x] = from_f<T>(0.f);
      Vc[base + x] = from_f<T>(0.f);
    }
  }
}

// len[i] += n_tok[i]; masked variant: layer_len[l][i] += n_tok[i] where the
// prompt executed layer l.
__global__ void pf_advance_kernel(int B, int L, const int32_t* n_tok, const uint8_t* mask, int32_t* len,
                                  int32_t* layer_len, int kv_batch, const int32_t* status) {
  if (call_aborted(status)) return;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B) return;
  const int t = n_tok[i];
  len[i] += t;
  if (layer_len != nullptr)
    for (int l = 0; l < L; ++l) layer_len[(size_t)l * kv_batch + i] += mask[(size_t)i * L + l] ? t : 0;
}

// ---------------------------------------------------------------------------
// One block over m prompt-token rows
// ---------------------------------------------------------------------------
struct PfLayerWork {
  const int32_t* rows;     // device [m] token rows, or nullptr (all tokens, identity)
  int m;
  const int4* items;       // device attention work items
  int n_items;
};

static void pf_block(Ctx& c, const buddy_kv_state& kv, int l, const PfLayerWork& w, const float* src, float* H,
                     cudaStream_t s, bool prof) {
  const buddy_layer_weights& W = c.layers[l];
  const bool split = l <= c.cl;   // blocks that feed the router keep ~16-bit activations
  const RowSel sel{w.rows, nullptr, w.m};
  const int32_t* base = cache_len(c, kv, l);
  {
    ProfScope p(c, s, BUDDY_PROF_PF_OTHER, 1, prof);
    launch_rmsnorm(c, src, sel, W.attn_norm, c.pf_xn, split ? c.pf_xn_lo : nullptr, s);
  }
  PfEpi e{};
  e.rows = w.rows;
  e.q_out = c.pf_q;
  e.bias = W.b_qkv;
  e.tok_seq = c.pf_tok_seq;
  e.tok_pos = c.pf_tok_pos;
  e.len = kv.len;
  e.cache_len = base;
  e.seq_off = kv.seq_off;
  e.cap = kv.cap;
  e.kc = kv.k_cache[l];
  e.vc = kv.v_cache[l];
  {
    ProfScope p(c, s, BUDDY_PROF_PF_GEMM, 1, prof);
    launch_gemm_pf(c, EPI_QKV, split, l, 0, 0, w.m, e, s);
  }
  {
    ProfScope p(c, s, BUDDY_PROF_PF_ATTENTION, 1, prof);
    launch_attention_pf(c, w.n_items, w.items, c.pf_n_tok, base, kv, l, c.pf_q, c.pf_attn,
                        split ? c.pf_attn_lo : nullptr, s);
  }
  e = PfEpi{};
  e.rows = w.rows;
  e.resid_src = src;
  e.resid_dst = H;
  {
    ProfScope p(c, s, BUDDY_PROF_PF_GEMM, 1, prof);
    launch_gemm_pf(c, EPI_RESID, split, l, 1, 1, w.m, e, s);
  }
  {
    ProfScope p(c, s, BUDDY_PROF_PF_OTHER, 1, prof);
    launch_rmsnorm(c, H, sel, W.ffn_norm, c.pf_xn, split ? c.pf_xn_lo : nullptr, s);
  }
  e = PfEpi{};
  e.out_act = c.pf_act;
  e.out_act_lo = split ? c.pf_act_lo : nullptr;
  {
    ProfScope p(c, s, BUDDY_PROF_PF_GEMM, 1, prof);
    launch_gemm_pf(c, EPI_SWIGLU, split, l, 2, 0, w.m, e, s);
  }
  e = PfEpi{};
  e.rows = w.rows;
  e.resid_src = H;
  e.resid_dst = H;
  {
    ProfScope p(c, s, BUDDY_PROF_PF_GEMM, 1, prof);
    launch_gemm_pf(c, EPI_RESID, split, l, 3, 2, w.m, e, s);
  }
}

// ---------------------------------------------------------------------------
// The call
// ---------------------------------------------------------------------------
int run_prefill(Ctx& c, const buddy_kv_state& kv, int B, const int32_t* n_tok_host, const float* x, const int32_t* k,
                float* h_out, uint8_t* mask_out, float* scores_out, cudaStream_t s) {
  const bool prof = c.profiling != 0;
  std::vector<int32_t> off(B + 1, 0);
  for (int i = 0; i < B; ++i) off[i + 1] = off[i] + n_tok_host[i];
  const int T = off[B];
  std::vector<int32_t> tok_seq(T), tok_t(T);
  for (int i = 0; i < B; ++i)
    for (int t = 0; t < n_tok_host[i]; ++t) {
      tok_seq[off[i] + t] = i;
      tok_t[off[i] + t] = t;
    }
  std::vector<int32_t> ends(off.begin() + 1, off.end());
#define PCK(x)                                                                             \
  do {                                                                                     \
    cudaError_t e_ = (x);                                                                  \
    if (e_ != cudaSuccess) {                                                               \
      fprintf(stderr, "libbuddy: prefill: %s -> %s\n", #x, cudaGetErrorString(e_));        \
      return BUDDY_ERR_CUDA;                                                               \
    }                                                                                      \
  } while (0)
  PCK(cudaMemcpyAsync(c.pf_tok_seq, tok_seq.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, s));
  PCK(cudaMemcpyAsync(c.pf_tok_t, tok_t.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, s));
  PCK(cudaMemcpyAsync(c.pf_n_tok, n_tok_host, sizeof(int32_t) * B, cudaMemcpyHostToDevice, s));
  PCK(cudaMemcpyAsync(c.pf_tok_end, ends.data(), sizeof(int32_t) * B, cudaMemcpyHostToDevice, s));
  const int k_min = c.have_pred ? 0 : 1;
  pf_check_kernel<<<1, 256, 0, s>>>(B, k, c.Lm, k_min, c.pf_n_tok, kv.len, kv.cap, c.max_pos,
                                    c.masked ? kv.layer_len : nullptr, c.L, kv.batch, c.status);
  pf_tokens_kernel<<<(T + 255) / 256, 256, 0, s>>>(T, c.pf_tok_seq, c.pf_tok_t, kv.len, c.pf_tok_pos, c.status);

  // attention work items for a set of sequences: 64 query tokens x one head
  auto items_for = [&](const std::vector<int>& seqs, std::vector<int4>& out) {
    int j = 0;
    for (int i : seqs) {
      for (int t0 = 0; t0 < n_tok_host[i]; t0 += 64)
        for (int h = 0; h < c.nq; ++h) out.push_back(make_int4(i, h, j + t0, t0));
      j += n_tok_host[i];
    }
  };
  std::vector<int> all(B);
  for (int i = 0; i < B; ++i) all[i] = i;
  std::vector<int4> items_all;
  items_for(all, items_all);
  if ((int64_t)items_all.size() > c.pf_items_max) return BUDDY_ERR_RANGE;
  // slot 0 of the item buffer: every sequence; slots 1.. : the routed layers
  PCK(cudaMemcpyAsync(c.pf_items, items_all.data(), sizeof(int4) * items_all.size(), cudaMemcpyHostToDevice, s));
  const PfLayerWork every{nullptr, T, c.pf_items, (int)items_all.size()};

  // blocks 0..c on every token, then the router per prompt
  for (int l = 0; l <= c.cl; ++l) pf_block(c, kv, l, every, l == 0 ? x : h_out, h_out, s, prof);
  {
    ProfScope p(c, s, BUDDY_PROF_ROUTE, 1, prof);
    launch_pool_refresh_n(c, kv, B, c.pf_n_tok, s);
    pf_gather_kernel<<<B, 256, 0, s>>>(B, c.d, c.pf_tok_end, h_out, kv.len, c.pf_n_tok, c.pf_hlast, c.pf_cnt,
                                       c.status);
    launch_route(c, B, c.pf_hlast, kv.pool_sum, c.pf_cnt, 0, k, c.mask, c.sel, c.scores, s);
  }
  // the routes come back to the host, which sizes every later launch
  std::vector<uint8_t> mask((size_t)B * c.L);
  int32_t st[2] = {0, 0};
  PCK(cudaMemcpyAsync(mask.data(), c.mask, mask.size(), cudaMemcpyDeviceToHost, s));
  PCK(cudaMemcpyAsync(st, c.status, sizeof(st), cudaMemcpyDeviceToHost, s));
  PCK(cudaStreamSynchronize(s));
  if (st[1] != 0) return BUDDY_ERR_DEVICE;   // checks failed: nothing was written

  if (!c.masked) {
    LayerPtrs p;
    for (int l = 0; l < c.L; ++l) {
      p.k[l] = kv.k_cache[l];
      p.v[l] = kv.v_cache[l];
    }
    ProfScope ps(c, s, BUDDY_PROF_PF_OTHER, 1, prof);
    dim3 g(std::max(1, c.Lm), B);
    if (c.dtype == BUDDY_DTYPE_BF16)
      pf_zero_kernel<bf16><<<g, 256, 0, s>>>(B, c.L, c.cl + 1, c.nkv, c.hd, c.mask, p, kv.len, c.pf_n_tok,
                                             kv.seq_off, kv.cap, c.status);
    else
      pf_zero_kernel<float><<<g, 256, 0, s>>>(B, c.L, c.cl + 1, c.nkv, c.hd, c.mask, p, kv.len, c.pf_n_tok,
                                              kv.seq_off, kv.cap, c.status);
  }
  // row lists and work items of the routed layers
  std::vector<int32_t> rows_all;
  std::vector<int4> items_l;
  std::vector<PfLayerWork> work(c.L);
  std::vector<size_t> row_at(c.L), item_at(c.L);
  for (int l = c.cl + 1; l < c.L - 1; ++l) {
    std::vector<int> seqs;
    for (int i = 0; i < B; ++i)
      if (mask[(size_t)i * c.L + l]) seqs.push_back(i);
    row_at[l] = rows_all.size();
    item_at[l] = items_l.size();
    for (int i : seqs)
      for (int t = off[i]; t < off[i + 1]; ++t) rows_all.push_back(t);
    items_for(seqs, items_l);
    work[l].m = (int)(rows_all.size() - row_at[l]);
    work[l].n_items = (int)(items_l.size() - item_at[l]);
  }
  if ((int64_t)rows_all.size() > (int64_t)c.L * c.pf_max || (int64_t)(items_l.size() + items_all.size()) >
                                                              (int64_t)(c.L + 1) * c.pf_items_max)
    return BUDDY_ERR_RANGE;
  if (!rows_all.empty())
    PCK(cudaMemcpyAsync(c.pf_rows, rows_all.data(), sizeof(int32_t) * rows_all.size(), cudaMemcpyHostToDevice, s));
  if (!items_l.empty())
    PCK(cudaMemcpyAsync(c.pf_items + items_all.size(), items_l.data(), sizeof(int4) * items_l.size(),
                        cudaMemcpyHostToDevice, s));
  for (int l = c.cl + 1; l < c.L - 1; ++l) {
    if (work[l].m == 0) continue;
    work[l].rows = c.pf_rows + row_at[l];
    work[l].items = c.pf_items + items_all.size() + item_at[l];
    pf_block(c, kv, l, work[l], h_out, h_out, s, prof);
  }
  pf_block(c, kv, c.L - 1, every, h_out, h_out, s, prof);
  {
    ProfScope p(c, s, BUDDY_PROF_PF_OTHER, 1, prof);
    pf_advance_kernel<<<(B + 255) / 256, 256, 0, s>>>(B, c.L, c.pf_n_tok, c.mask, kv.len,
                                                      c.masked ? kv.layer_len : nullptr, kv.batch, c.status);
  }
  if (mask_out) PCK(cudaMemcpyAsync(mask_out, c.mask, (size_t)B * c.L, cudaMemcpyDeviceToDevice, s));
  if (scores_out)
    PCK(cudaMemcpyAsync(scores_out, c.scores, (size_t)B * c.Lm * sizeof(float), cudaMemcpyDeviceToDevice, s));
  PCK(cudaGetLastError());
#undef PCK
  return BUDDY_OK;
}

}  // namespace buddy

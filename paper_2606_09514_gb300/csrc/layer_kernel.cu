// One executed decoder block (Eq. 1, executed branch) as a single persistent
// cooperative kernel, for small batches (every active row fits one 16-column
// MMA tile).  Decode at small batch is bound by streaming the layer's weights;
// separate kernels leave HBM idle between launches (ramp-up, tails, launch
// latency).  Here one CTA per SM runs the whole block as phases separated by
// grid-wide barriers:
//
//   norm1 | B1 | QKV GEMM (+bias, RoPE, cache append, pool) | B2 | attention |
//   B3 | O GEMM (+residual) | B4 | norm2 | B5 | gate/up GEMM (+SwiGLU) | B6 |
//   down GEMM (+residual)
//
// Warp 0 streams the weight tiles of all four GEMMs, in order, through one
// shared-memory ring without waiting for the barriers: an activation tile is
// added to a stage only once the barrier that makes those activations ready
// has passed, so weight traffic continues while the other warps cross
// barriers, normalise or attend.  Warp 1 issues tcgen05 MMAs; warps 2-5 run the
// epilogues, the normalisations and the attention, and the grid barriers.
// Every wait is bounded (global timer); a timeout raises BUDDY_DEV_TIMEOUT and
// the kernel drains its copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "attn_common.cuh"
#include "common.cuh"
#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace buddy {

constexpr int kLkThreads = 192;

struct LkMaps {
  CUtensorMap w[4];     // qkv, o, gate_up, down weights
  CUtensorMap x[4];     // activation operand of each GEMM (xn, attn, xn, act)
  CUtensorMap xlo[4];   // remainder terms (first layer)
};

struct LkParams {
  const int32_t* rows;
  const int32_t* count;
  int n;
  const float* src;      // residual input of the block (h_in for the first layer)
  float* H;              // residual output, updated in place for the block's rows
  const float* g1;
  const float* g2;
  float eps;
  int d;
  bf16* xn;
  bf16* xn_lo;
  int stages;
  uint32_t stage_bytes;
  uint32_t tmem_cols;
  uint32_t attn_off;     // byte offset of the attention region in dynamic shared memory
  unsigned* bar;         // grid barrier: [0] arrivals, [1] generation
  TcParams tp[4];        // epilogue parameters of each GEMM
  AttnArgs<bf16> attn;
  int attn_gp;           // padded query heads per KV head (attention template)
  int32_t* status;
};

// Barrier count after which each GEMM's activation operand is ready.
__device__ __forceinline__ int x_ready(int ph) { return ph == 0 ? 1 : (ph == 1 ? 3 : (ph == 2 ? 5 : 6)); }

// ---------------------------------------------------------------------------
// Grid barrier among the epilogue warps of all CTAs (sense by generation).
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool lk_grid_sync(unsigned* bar, unsigned& gen, volatile int* abort_flag,
                                             volatile int* passed, volatile int* ok_s, const int32_t* status) {
  asm volatile("fence.proxy.async.global;" ::: "memory");   // generic writes -> later TMA reads
  epi_bar();
  if (threadIdx.x == 64) {
    bool ok = !*abort_flag;
    if (ok) {
      __threadfence();
      const unsigned g = gen;
      const unsigned arrived = atomicAdd(&bar[0], 1u);
      if (arrived == gridDim.x - 1) {
        bar[0] = 0;
        __threadfence();
        atomicExch(&bar[1], g + 1);
      } else {
        const uint64_t t0 = ptx::globaltimer();
        while (*reinterpret_cast<volatile unsigned*>(&bar[1]) == g) {
          if (*reinterpret_cast<const volatile int32_t*>(status + 1) != 0 ||
              ptx::globaltimer() - t0 > kWaitLimitNs) {
            ok = false;
            break;
          }
        }
      }
      __threadfence();
      gen = g + 1;
    }
    if (!ok) *abort_flag = 1;
    *ok_s = ok;
    if (ok) *passed = *passed + 1;
  }
  epi_bar();
  return *ok_s != 0;
}

// RMSNorm of the block's rows, 32 columns per CTA: xn = bf16(x * rsqrt(mean(x^2) + eps) * g)
// (plus the remainder term with SPLIT).  128 epilogue threads, t = 0..127.
template <bool SPLIT>
__device__ __forceinline__ void lk_norm(const LkParams& p, const float* X, const float* gam, int m, int t,
                                        float* red, float* inv) {
  const int nch = p.d / 32;
  if ((int)blockIdx.x >= nch) return;
  for (int j = 0; j < m; ++j) {
    const float* x = X + (size_t)(p.rows ? p.rows[j] : j) * p.d;
    float ss = 0.f;
    for (int e = t * 4; e < p.d; e += 512) {
      const float4 v = *reinterpret_cast<const float4*>(x + e);
      ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = warp_sum(ss);
    if ((t & 31) == 0) red[j * 4 + (t >> 5)] = ss;
  }
  epi_bar();
  if (t < m) inv[t] = rsqrtf((red[t * 4] + red[t * 4 + 1] + red[t * 4 + 2] + red[t * 4 + 3]) / (float)p.d + p.eps);
  epi_bar();
  for (int c = blockIdx.x; c < nch; c += gridDim.x) {
    for (int x = t; x < m * 32; x += 128) {
      const int j = x >> 5, e = c * 32 + (x & 31);
      const float y = X[(size_t)(p.rows ? p.rows[j] : j) * p.d + e] * inv[j] * gam[e];
      const bf16 hi = from_f<bf16>(y);
      p.xn[(size_t)j * p.d + e] = hi;
      if (SPLIT) p.xn_lo[(size_t)j * p.d + e] = from_f<bf16>(y - to_f(hi));
    }
  }
}

// Drains this CTA's units of GEMM `ph` from TMEM and applies its epilogue.
template <int EPI, bool SPLIT>
__device__ __forceinline__ bool lk_epilogue(const LkParams& p, int ph, int m, uint32_t tmem_base,
                                            uint64_t* tfull_bar, uint64_t* tempty_bar, int& acc, uint32_t& acc_ph,
                                            volatile int* abort_flag, int* last_flag) {
  const TcParams& tp = p.tp[ph];
  const uint32_t acc_cols = (uint32_t)(tp.mt * tp.bw);
  for (int u = blockIdx.x; u < tp.units; u += gridDim.x) {
    const bool ok = ptx::mbar_wait_bounded(&tfull_bar[acc], acc_ph, kWaitLimitNs, abort_flag);
    if (epi_bar_any(!ok)) return false;
    ptx::tc_fence_after();
    tc_epilogue_unit<EPI, SPLIT>(tp, u, m, tmem_base + (uint32_t)acc * acc_cols, &tempty_bar[acc], last_flag);
    acc ^= 1;
    if (acc == 0) acc_ph ^= 1u;
  }
  return true;
}

template <bool SPLIT>
__global__ void __launch_bounds__(kLkThreads, 1)
    layer_kernel(const __grid_constant__ LkMaps maps, const LkParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kTcMaxStages], empty_bar[kTcMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag, passed, ok_s, consumed;
  __shared__ int last_flag;
  __shared__ float red[64], inv[16], sc[32];

  if (call_aborted(p.status)) return;
  const int m = p.count ? *p.count : p.n;
  if (m <= 0) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      ptx::mbar_init(&full_bar[s], 1);
      ptx::mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&tfull_bar[a], 1);
      ptx::mbar_init(&tempty_bar[a], 4);
    }
    ptx::mbar_init(&done_bar, 1);
    abort_flag = 0;
    passed = 0;
    consumed = 0;
    ptx::fence_mbar_init();
    for (int w = 0; w < 4; ++w) ptx::tma_prefetch_desc(&maps.w[w]);
  }
  if (warp == 1) {
    ptx::tmem_alloc(&tmem_slot, p.tmem_cols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = tmem_slot;
  const uint32_t x_bytes = tc_x_bytes(m, SPLIT);
  const uint32_t w_bytes = (uint32_t)p.tp[0].bw * 128u;

  if (warp == 0) {
    // --------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t pol = ptx::policy_evict_first();
      int pend_stage[kTcMaxStages] = {}, pend_ph[kTcMaxStages] = {}, pend_kb[kTcMaxStages] = {};
      int ph_head = 0, ph_cnt = 0;
      auto flush = [&]() {
        while (ph_cnt > 0 && passed >= x_ready(pend_ph[ph_head])) {
          const int s = pend_stage[ph_head], ph = pend_ph[ph_head], kb = pend_kb[ph_head];
          ptx::mbar_arrive_expect_tx(&full_bar[s], x_bytes);
          tc_load_x<SPLIT>(smem + (size_t)s * p.stage_bytes, &maps.x[ph], &maps.xlo[ph], &full_bar[s], p.tp[ph], m,
                           kb);
          ph_head = (ph_head + 1) % kTcMaxStages;
          --ph_cnt;
        }
      };
      int stage = 0, issued = 0;
      uint32_t ph_bit = 0;
      bool ok = true;
      for (int ph = 0; ph < 4 && ok; ++ph) {
        const TcParams& G = p.tp[ph];
        for (int u = blockIdx.x; u < G.units && ok; u += gridDim.x) {
          const int tile = u % G.n_tiles, split = u / G.n_tiles;
          const int kb0 = split * G.kb_per_split, kb1 = min(G.kb_total, kb0 + G.kb_per_split);
          for (int kb = kb0; kb < kb1; ++kb) {
            // a free slot; meanwhile activation tiles whose barrier passed go out
            const uint64_t t0 = ptx::globaltimer();
            while (true) {
              flush();
              if (ptx::mbar_try_wait(&empty_bar[stage], ph_bit ^ 1u)) break;
              if (abort_flag || ptx::globaltimer() - t0 > kWaitLimitNs) {
                abort_flag = 1;
                ok = false;
                break;
              }
            }
            if (!ok) break;
            uint8_t* a = smem + (size_t)stage * p.stage_bytes;
            // activations already available (no earlier stage waiting): one
            // arrival covers both tiles; otherwise the activation tile waits
            // in the queue for its barrier
            const bool x_now = ph_cnt == 0 && passed >= x_ready(ph);
            if (x_now) ptx::mbar_arrive_expect_tx(&full_bar[stage], w_bytes + x_bytes);
            else ptx::mbar_expect_tx(&full_bar[stage], w_bytes);
            if (ph == 2) tc_load_w<EPI_SWIGLU>(a, &maps.w[2], &full_bar[stage], G, tile, kb, pol);
            else tc_load_w<EPI_RESID>(a, &maps.w[ph], &full_bar[stage], G, tile, kb, pol);
            if (x_now) {
              tc_load_x<SPLIT>(a, &maps.x[ph], &maps.xlo[ph], &full_bar[stage], G, m, kb);
            } else {
              const int slot = (ph_head + ph_cnt) % kTcMaxStages;
              pend_stage[slot] = stage;
              pend_ph[slot] = ph;
              pend_kb[slot] = kb;
              ++ph_cnt;
              flush();
            }
            ++issued;
            if (++stage == p.stages) {
              stage = 0;
              ph_bit ^= 1u;
            }
          }
        }
      }
      // the last activation tiles go out once their barrier passes
      const uint64_t t0 = ptx::globaltimer();
      while (ok && ph_cnt > 0) {
        flush();
        if (abort_flag || ptx::globaltimer() - t0 > kWaitLimitNs) {
          abort_flag = 1;
          break;
        }
      }
      // never leave with copies in flight: every stage whose activation tile
      // was issued must land; stages still waiting for one get their arrival
      for (int k = 0; k < ph_cnt; ++k) ptx::mbar_arrive(&full_bar[pend_stage[(ph_head + k) % kTcMaxStages]]);
      for (int it = consumed; it < issued; ++it) {
        volatile int dummy = 0;
        ptx::mbar_wait_bounded(&full_bar[it % p.stages], (uint32_t)((it / p.stages) & 1), kWaitLimitNs, &dummy);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = ptx::idesc_bf16(128u, (uint32_t)p.tp[0].bw);
      int stage = 0, acc = 0, n_consumed = 0;
      uint32_t ph_bit = 0, acc_ph = 0;
      bool ok = true;
      for (int ph = 0; ph < 4 && ok; ++ph) {
        const TcParams& G = p.tp[ph];
        for (int u = blockIdx.x; u < G.units && ok; u += gridDim.x) {
          const int split = u / G.n_tiles;
          const int kb0 = split * G.kb_per_split, kb1 = min(G.kb_total, kb0 + G.kb_per_split);
          if (!ptx::mbar_wait_bounded(&tempty_bar[acc], acc_ph ^ 1u, kWaitLimitNs, &abort_flag)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t dcol = tmem_base + (uint32_t)(acc * G.mt * G.bw);
          for (int kb = kb0; kb < kb1; ++kb) {
            if (!ptx::mbar_wait_bounded(&full_bar[stage], ph_bit, kWaitLimitNs, &abort_flag)) {
              ok = false;
              break;
            }
            consumed = ++n_consumed;
            ptx::tc_fence_after();
            tc_mma_stage<SPLIT>(smem + (size_t)stage * p.stage_bytes, dcol, G, m, idesc, kb == kb0);
            ptx::mma_commit(&empty_bar[stage]);
            if (++stage == p.stages) {
              stage = 0;
              ph_bit ^= 1u;
            }
          }
          if (!ok) break;
          ptx::mma_commit(&tfull_bar[acc]);
          acc ^= 1;
          if (acc == 0) acc_ph ^= 1u;
        }
      }
      ptx::mma_commit(&done_bar);
      volatile int dummy = 0;
      ptx::mbar_wait_bounded(&done_bar, 0, kWaitLimitNs, &dummy);
    }
    __syncwarp();
  } else {
    // ----------------------------------------- epilogue warps: phase program
    const int t = threadIdx.x - 64;
    unsigned gen = *reinterpret_cast<volatile unsigned*>(&p.bar[1]);
    int acc = 0;
    uint32_t acc_ph = 0;
    bool ok = true;
    lk_norm<SPLIT>(p, p.src, p.g1, m, t, red, inv);
    ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                          // B1
    if (ok) ok = lk_epilogue<EPI_QKV, SPLIT>(p, 0, m, tmem_base, tfull_bar, tempty_bar, acc, acc_ph, &abort_flag,
                                              &last_flag);
    if (ok) ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                  // B2
    if (ok) {
      uint8_t* as = smem + p.attn_off;
      switch (p.attn_gp) {
        case 1: attn_run<bf16, 128, 1, 128>(p.attn, t, blockIdx.x, gridDim.x, as, sc, SyncEpilogueWarps{}, false); break;
        case 2: attn_run<bf16, 128, 2, 128>(p.attn, t, blockIdx.x, gridDim.x, as, sc, SyncEpilogueWarps{}, false); break;
        case 4: attn_run<bf16, 128, 4, 128>(p.attn, t, blockIdx.x, gridDim.x, as, sc, SyncEpilogueWarps{}, false); break;
        default: attn_run<bf16, 128, 8, 128>(p.attn, t, blockIdx.x, gridDim.x, as, sc, SyncEpilogueWarps{}, false);
      }
      ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                        // B3
    }
    if (ok) ok = lk_epilogue<EPI_RESID, SPLIT>(p, 1, m, tmem_base, tfull_bar, tempty_bar, acc, acc_ph, &abort_flag,
                                              &last_flag);
    if (ok) ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                  // B4
    if (ok) {
      lk_norm<SPLIT>(p, p.H, p.g2, m, t, red, inv);
      ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                        // B5
    }
    if (ok) ok = lk_epilogue<EPI_SWIGLU, SPLIT>(p, 2, m, tmem_base, tfull_bar, tempty_bar, acc, acc_ph, &abort_flag,
                                              &last_flag);
    if (ok) ok = lk_grid_sync(p.bar, gen, &abort_flag, &passed, &ok_s, p.status);                  // B6
    if (ok) ok = lk_epilogue<EPI_RESID, SPLIT>(p, 3, m, tmem_base, tfull_bar, tempty_bar, acc, acc_ph, &abort_flag,
                                              &last_flag);
    if (!ok && t == 0) abort_flag = 1;
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (threadIdx.x == 0 && abort_flag) {
    atomicOr(p.status, BUDDY_DEV_TIMEOUT);
    atomicExch(p.status + 1, 1);
  }
  if (warp == 1) ptx::tmem_dealloc(tmem_base, p.tmem_cols);
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
// Ring of stages followed by the attention region.
constexpr int kLkSmemLimit = 227 * 1024 - 2 * 1024;   // room for static shared memory

static int lk_smem_budget(const Ctx& c, bool split, size_t attn_bytes, int* stages, uint32_t* stage_bytes) {
  const uint32_t sb = c.tc_stage_bytes[split ? 1 : 0];
  const int tail = (int)((attn_bytes + 1023) & ~size_t(1023));
  const int avail = kLkSmemLimit - 1024 - tail;
  *stages = std::min(kTcMaxStages, avail / (int)sb);
  *stage_bytes = sb;
  return *stages >= 3 ? (int)(*stages * sb + 1024 + tail) : 0;
}

bool layer_kernel_supported(const Ctx& c) {
  return c.use_tc && c.tc_mt == 1 && c.maxB <= 16 && c.hd == 128 && c.d % 32 == 0 && c.nq / c.nkv <= 8;
}

// One block on the rows of `sel` with the persistent kernel.  Returns false if
// the launch could not be made (the caller then uses the separate kernels).
bool launch_layer_kernel(const Ctx& c, const buddy_kv_state& kv, int l, RowSel sel, const float* src, float* H,
                         cudaStream_t s) {
  const bool split = c.split0 && l == 0;
  const int G = c.nq / c.nkv;
  const size_t attn_bytes = attn_smem_bytes(attn_smem_fixed<bf16, 128>(), G, 128, c.attn_max_chunks, c.maxB);
  int stages;
  uint32_t stage_bytes;
  const int smem = lk_smem_budget(c, split, attn_bytes, &stages, &stage_bytes);
  if (smem == 0) return false;
  static bool attr_set[2] = {false, false};
  if (!attr_set[split]) {
    if (cudaFuncSetAttribute(split ? layer_kernel<true> : layer_kernel<false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, kLkSmemLimit) != cudaSuccess)
      return false;
    attr_set[split] = true;
  }
  const buddy_layer_weights& W = c.layers[l];
  LkMaps maps;
  for (int w = 0; w < 4; ++w) maps.w[w] = c.tmaps_host[(size_t)l * 4 + w];
  const CUtensorMap* X = &c.tmaps_host[(size_t)c.L * 4];
  maps.x[0] = X[0]; maps.x[1] = X[1]; maps.x[2] = X[0]; maps.x[3] = X[2];
  maps.xlo[0] = X[3]; maps.xlo[1] = X[4]; maps.xlo[2] = X[3]; maps.xlo[3] = X[5];
  LkParams p{};
  p.rows = sel.rows; p.count = sel.count; p.n = sel.n;
  p.src = src; p.H = H; p.g1 = W.attn_norm; p.g2 = W.ffn_norm; p.eps = c.cfg.rms_eps; p.d = c.d;
  p.xn = (bf16*)c.xn; p.xn_lo = (bf16*)c.xn_lo;
  for (int w = 0; w < 4; ++w) {
    int N, K, tiles;
    gemm_shape(c, w, &N, &K, &tiles);
    TcParams& tp = p.tp[w];
    tp.N = N; tp.K = K; tp.n_tiles = tiles; tp.splits = c.tc_splits[w];
    tp.kb_total = (K + kTileK - 1) / kTileK;
    tp.kb_per_split = (tp.kb_total + tp.splits - 1) / tp.splits;
    tp.units = tiles * tp.splits;
    tp.bw = c.tc_bw; tp.mt = c.tc_mt; tp.rows_max = c.tc_rows_max; tp.stages = stages; tp.acc_bufs = 2;
    tp.stage_bytes = stage_bytes; tp.xr = c.tc_xr; tp.w_off = c.tc_w_off[split ? 1 : 0]; tp.tmem_cols = 512;
    tp.rows = sel.rows; tp.count = sel.count; tp.n = sel.n;
    tp.ws = c.gemm_ws; tp.ctr = c.gemm_ctr; tp.status = c.status;
  }
  TcParams& q = p.tp[0];   // QKV: fused finalisation
  q.bias = W.b_qkv; q.rope_cos = c.rope_cos; q.rope_sin = c.rope_sin; q.len = kv.len; q.seq_off = kv.seq_off;
  q.cap = kv.cap; q.kc = (bf16*)kv.k_cache[l]; q.vc = (bf16*)kv.v_cache[l]; q.q_out = c.q;
  q.pool = l == 0 ? kv.pool_sum : nullptr; q.nq = c.nq; q.nkv = c.nkv; q.hd = c.hd;
  p.tp[1].resid_src = src; p.tp[1].resid_dst = H;
  p.tp[2].out_act = (bf16*)c.act; p.tp[2].out_act_lo = split ? (bf16*)c.act_lo : nullptr;
  p.tp[3].resid_src = H; p.tp[3].resid_dst = H;
  p.stages = stages; p.stage_bytes = stage_bytes; p.tmem_cols = 512;   // one CTA per SM, two accumulators
  p.attn_off = (uint32_t)(stages * stage_bytes);
  p.bar = c.lk_bar;
  p.attn = AttnArgs<bf16>{c.q, sel.rows, sel.count, sel.n, c.nq, c.nkv, kv.len, kv.seq_off, kv.cap,
                          (const bf16*)kv.k_cache[l], (const bf16*)kv.v_cache[l], c.attn_max_chunks, c.attn_m,
                          c.attn_l, c.attn_acc, c.attn_ctr, (bf16*)c.attn_out, split ? (bf16*)c.attn_lo : nullptr,
                          c.status};
  p.attn_gp = attn_group_pad(G);
  p.status = c.status;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(c.num_sms);
  cfg.blockDim = dim3(kLkThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = split ? cudaLaunchKernelEx(&cfg, layer_kernel<true>, maps, p)
                              : cudaLaunchKernelEx(&cfg, layer_kernel<false>, maps, p);
  return e == cudaSuccess;
}

}  // namespace buddy

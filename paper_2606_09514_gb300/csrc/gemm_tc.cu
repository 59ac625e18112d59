// Tensor-core GEMM for the bf16 decode projections on sm_103a.
//
//   C[j][n] = sum_k X[j][k] * W[n][k]      (j < m active rows, n < N features)
//
// Decode GEMMs are skinny (m = 1..256) and bound by streaming W from HBM.  The
// tile geometry, the ring stage layout and the epilogues are described in
// gemm_common.cuh.  Persistent CTAs (one per SM) walk work units (weight tile,
// K split); warp 0 issues TMA loads into a ring of stages, warp 1 issues the
// tcgen05 MMAs (accumulating fp32 in TMEM), warps 2-5 drain TMEM and run the
// epilogue.  A tile split over K is finished by the last CTA to arrive, which
// sums the partials in split order (deterministic).
//
// Epilogues: fp32 store; residual add into the (row-gathered) hidden state;
// SwiGLU (a tile holds 128 gate rows and the matching 128 up rows); QKV
// finalisation (bias, RoPE, q, K/V cache append, pooled first-layer V).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>

#include "common.cuh"
#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace buddy {

// SPLIT: the activations are given as two bf16 terms hi + lo (hi = bf16(x),
// lo = bf16(x - hi)); every K step issues one MMA per term into the same
// accumulator, so the product carries ~16 mantissa bits of the activations.
template <int EPI, bool SPLIT>
__global__ void __launch_bounds__(kTcThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tx,
                   const __grid_constant__ CUtensorMap txlo, const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kTcMaxStages], empty_bar[kTcMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2], done_bar, pfull_bar[2];
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ volatile int consumed;
  __shared__ int last_flag;
  __shared__ float pred[32], pinv[8];   // panel mode: sums of squares, 1 / rms per row
  __shared__ int prow[8];               // panel mode: source row of each panel row

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  // A layer that no row selected leaves before any setup.  Its row count was
  // written by the compaction kernel; unless that kernel is the one enqueued
  // right before this GEMM (count_late), it completed before the preceding
  // kernel let this one launch (every kernel of the step waits on its
  // predecessor before allowing its dependents to start), so the count may be
  // read before the wait.  The wait itself always happens, so that the
  // completion of this kernel implies the completion of everything enqueued
  // before it.
  bool waited = false;
  if (p.count_late) {
    pdl_wait();
    waited = true;
  }
  if (p.count && *reinterpret_cast<const volatile int32_t*>(p.count) <= 0) {
    if (!waited) pdl_wait();
    pdl_trigger();
    return;
  }

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
    ptx::mbar_init(&pfull_bar[0], 1);
    ptx::mbar_init(&pfull_bar[1], 1);
    abort_flag = 0;
    consumed = 0;
    ptx::fence_mbar_init();
    ptx::tma_prefetch_desc(&tw);
    ptx::tma_prefetch_desc(&tx);
    if (SPLIT) ptx::tma_prefetch_desc(&txlo);
  }
  if (warp == 1) {
    ptx::tmem_alloc(&tmem_slot, p.tmem_cols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = tmem_slot;
  const uint32_t w_bytes = (uint32_t)p.bw * 128u;

  // Weight tiles depend on nothing an earlier kernel writes: start streaming
  // the first `stages` of them before waiting for the predecessor.
  int npre = 0;
  uint64_t pol = 0;
  if (warp == 0 && lane == 0) {
    pol = ptx::policy_evict_first();
    for (int u = blockIdx.x; u < p.units && npre < p.stages; u += gridDim.x) {
      const int tile = u % p.n_tiles, split = u / p.n_tiles;
      const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
      for (int kb = kb0; kb < kb1 && npre < p.stages; ++kb, ++npre) {
        ptx::mbar_expect_tx(&full_bar[npre], w_bytes);
        tc_load_w<EPI>(smem + (size_t)npre * p.stage_bytes, &tw, &full_bar[npre], p, tile, kb, pol);
      }
    }
  }
  const bool panel = p.nsrc != nullptr;
  const bool first_pass = panel && p.K <= kPanelFirstMaxK;
  if (first_pass && warp >= 2 && blockIdx.x < p.units) {
    // Before the wait: the RMSNorm gains of the first unit's K range (weights,
    // written by no kernel of the step) into shared memory, and the source
    // rows (written by the compaction kernel, complete before this kernel
    // could launch unless count_late, in which case the wait is behind us).
    const int et = threadIdx.x - 64;
    const int split = blockIdx.x / p.n_tiles;
    const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
    float* gst = reinterpret_cast<float*>(smem + p.gstage_off);
    for (int c = et * 4; c < (kb1 - kb0) * kTileK; c += 128 * 4)
      *reinterpret_cast<float4*>(gst + c) = *reinterpret_cast<const float4*>(p.ngamma + kb0 * kTileK + c);
    if (et < 8 && et < p.n) prow[et] = p.rows ? p.rows[et] : et;
  }
  if (!waited) pdl_wait();
  pdl_trigger();
  const int m = call_aborted(p.status) ? 0 : (p.count ? *p.count : p.n);
  if (m <= 0) {
    // nothing to compute: let the prefetched tiles land before leaving
    if (warp == 0 && lane == 0) {
      for (int it = 0; it < npre; ++it) {
        ptx::mbar_arrive(&full_bar[it]);
        volatile int dummy = 0;
        ptx::mbar_wait_bounded(&full_bar[it], 0, kWaitLimitNs, &dummy);
      }
    }
    __syncwarp();
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem_base, p.tmem_cols);
    return;
  }
  const uint32_t x_bytes = panel ? 0u : tc_x_bytes(m, SPLIT);
  const uint32_t acc_cols = (uint32_t)(p.mt * p.bw);

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
        const int tile = u % p.n_tiles, split = u / p.n_tiles;
        const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
        for (int kb = kb0; kb < kb1; ++kb) {
          uint8_t* st = smem + (size_t)stage * p.stage_bytes;
          if (issued < npre) {
            // weight tile already in flight: add the activation tiles
            if (panel) ptx::mbar_arrive(&full_bar[stage]);
            else ptx::mbar_arrive_expect_tx(&full_bar[stage], x_bytes);
          } else {
            if (!ptx::mbar_wait_bounded(&empty_bar[stage], ph ^ 1u, p.wait_ns, &abort_flag)) {
              ok = false;
              break;
            }
            ptx::mbar_arrive_expect_tx(&full_bar[stage], w_bytes + x_bytes);
            tc_load_w<EPI>(st, &tw, &full_bar[stage], p, tile, kb, pol);
          }
          if (!panel) tc_load_x<SPLIT>(st, &tx, &txlo, &full_bar[stage], p, m, kb);
          ++issued;
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1u;
          }
        }
      }
      // never leave with copies in flight: wait for every issued stage to land
      for (int it = consumed; it < issued; ++it) {
        volatile int dummy = 0;
        ptx::mbar_wait_bounded(&full_bar[it % p.stages], (uint32_t)((it / p.stages) & 1), kWaitLimitNs, &dummy);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA
    if (lane == 0) {
      const uint32_t idesc = ptx::idesc_bf16(128u, (uint32_t)p.bw);
      int stage = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      int n_consumed = 0, ui = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x, ++ui) {
        const int split = u / p.n_tiles;
        const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
        if (!ptx::mbar_wait_bounded(&tempty_bar[acc], acc_ph ^ 1u, p.wait_ns, &abort_flag)) break;
        if (panel &&
            !ptx::mbar_wait_bounded(&pfull_bar[ui & 1], (uint32_t)((ui >> 1) & 1), p.wait_ns, &abort_flag))
          break;
        ptx::tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)acc * acc_cols;
        const uint8_t* pan = smem + p.panel_off + (size_t)(ui & 1) * p.panel_bytes;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!ptx::mbar_wait_bounded(&full_bar[stage], ph, p.wait_ns, &abort_flag)) {
            ok = false;
            break;
          }
          consumed = ++n_consumed;
          ptx::tc_fence_after();
          if (panel)
            tc_mma_panel<SPLIT>(smem + (size_t)stage * p.stage_bytes, pan + (size_t)(kb - kb0) * 1024, d, p, idesc,
                                kb == kb0);
          else
            tc_mma_stage<SPLIT>(smem + (size_t)stage * p.stage_bytes, d, p, m, idesc, kb == kb0);
          ptx::mma_commit(&empty_bar[stage]);
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        ptx::mma_commit(&tfull_bar[acc]);
        if (p.acc_bufs == 2) {
          acc ^= 1;
          if (acc == 0) acc_ph ^= 1u;
        } else {
          acc_ph ^= 1u;
        }
      }
      // all issued MMAs complete before TMEM is released
      ptx::mma_commit(&done_bar);
      volatile int dummy = 0;
      ptx::mbar_wait_bounded(&done_bar, 0, kWaitLimitNs, &dummy);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- epilogue
    int acc = 0;
    uint32_t acc_ph = 0;
    const int et = threadIdx.x - 64;
    if (panel && blockIdx.x < p.units) {
      // the first unit's panel (and the norm of every row)
      const int split = blockIdx.x / p.n_tiles;
      const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
      if (first_pass) {
        epi_bar();   // staged gains and rows visible to all epilogue warps
        tc_panel_first<SPLIT>(p, smem + p.panel_off, m, kb0, kb1, et, prow,
                              reinterpret_cast<const float*>(smem + p.gstage_off), pred, pinv);
      } else {
        tc_panel_inv(p, m, et, pred, pinv);
        tc_panel_write<SPLIT>(p, smem + p.panel_off, m, kb0, kb1, et, pinv);
      }
      epi_bar();
      if (et == 0) ptx::mbar_arrive(&pfull_bar[0]);
    }
    int ui = 0;
    for (int u = blockIdx.x; u < p.units; u += gridDim.x, ++ui) {
      const int un = u + gridDim.x;
      if (panel && un < p.units) {
        // the next unit's panel goes into the buffer the unit before this one
        // used (its MMAs completed: its accumulator was drained)
        const int split = un / p.n_tiles;
        const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
        tc_panel_write<SPLIT>(p, smem + p.panel_off + (size_t)((ui + 1) & 1) * p.panel_bytes, m, kb0, kb1, et,
                              pinv);
        epi_bar();
        if (et == 0) ptx::mbar_arrive(&pfull_bar[(ui + 1) & 1]);
      }
      const bool ok = ptx::mbar_wait_bounded(&tfull_bar[acc], acc_ph, p.wait_ns, &abort_flag);
      if (epi_bar_any(!ok)) break;
      ptx::tc_fence_after();
      tc_epilogue_unit<EPI, SPLIT>(p, u, m, tmem_base + (uint32_t)acc * acc_cols, &tempty_bar[acc], &last_flag);
      if (p.acc_bufs == 2) {
        acc ^= 1;
        if (acc == 0) acc_ph ^= 1u;
      } else {
        acc_ph ^= 1u;
      }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (threadIdx.x == 0 && abort_flag) atomicOr(p.status, BUDDY_DEV_TIMEOUT);
  if (warp == 1) ptx::tmem_dealloc(tmem_base, p.tmem_cols);
}

// Deferred fixup of a GEMM whose units only staged their partials: items
// (tile, row, 4-column group) over the whole grid, each summing its splits in
// split order (the same order, hence the same result, as the in-kernel
// finisher) and applying the epilogue.  With row-major slots consecutive
// threads take consecutive groups of a row; with group-major slots a warp
// takes 8 rows x 4 groups (128 contiguous bytes of each group's partials,
// 4 contiguous groups of each row's outputs).
template <int EPI, bool SPLIT>
__global__ void __launch_bounds__(kTcFixThreads) gemm_fix_kernel(const TcParams p) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(p.status)) return;
  const int m = p.count ? *p.count : p.n;
  if (m <= 0) return;
  const int ng = tc_groups<EPI>(p);
  const long long stride = (long long)gridDim.x * kTcFixThreads;
  if (p.rows_max <= 16) {
    const long long items = (long long)p.n_tiles * m * ng;
    for (long long it = (long long)blockIdx.x * kTcFixThreads + threadIdx.x; it < items; it += stride) {
      const int g = (int)(it % ng);
      const long long r = it / ng;
      const int j = (int)(r % m), tile = (int)(r / m);
      tc_fix_item<EPI, SPLIT>(p, tile, j, tc_group_col<EPI>(p, g));
    }
  } else {
    // warp blocks of 8 rows x 4 groups (ng is a multiple of 4)
    const int rb = (m + 7) >> 3, gb = ng >> 2;
    const long long items = (long long)p.n_tiles * gb * rb * 32;
    const int lane = threadIdx.x & 31;
    for (long long it = (long long)blockIdx.x * kTcFixThreads + threadIdx.x; it < items; it += stride) {
      const long long wb = it >> 5;
      const int j = (int)(wb % rb) * 8 + (lane & 7);
      const long long r = wb / rb;
      const int g = (int)(r % gb) * 4 + (lane >> 3), tile = (int)(r / gb);
      if (j < m) tc_fix_item<EPI, SPLIT>(p, tile, j, tc_group_col<EPI>(p, g));
    }
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
typedef CUresult (*PFN_encodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                    const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                    CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static PFN_encodeTiled get_encode() {
  static PFN_encodeTiled fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_encodeTiled>(p);
  }
  return fn;
}

// 2-D bf16 map over a row-major [rows, K] matrix, box [64 cols, box_rows].
static bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows) {
  PFN_encodeTiled enc = get_encode();
  if (!enc) return false;
  const cuuint64_t dims[2] = {K, rows};
  const cuuint64_t strides[1] = {K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kTileK, box_rows};
  const cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Split-K factor.  Every SM streams at most its share of HBM bandwidth, so
// the units (tile, split) should keep all SMs busy: among the factors whose
// persistent waves are at least 90% occupied (every split >= 4 K blocks, none
// empty), the one with the fewest waves, then the fewest splits; otherwise the
// best occupancy.
static int choose_splits(int tiles, int kb, int sms) {
  int best = 1, best_waves = 1 << 30;
  double best_eff = -1.0;
  int fb = 1;
  double fb_eff = -1.0;
  for (int s = 1; s <= 16; ++s) {
    const int kps = (kb + s - 1) / s;
    if (s > 1 && (kps < 4 || (s - 1) * kps >= kb)) continue;
    const int units = tiles * s;
    const int waves = (units + sms - 1) / sms;
    const double eff = (double)units / (double)(waves * sms);
    if (eff >= 0.9 && waves < best_waves) {
      best = s;
      best_waves = waves;
      best_eff = eff;
    }
    if (eff > fb_eff + 0.02) {
      fb_eff = eff;
      fb = s;
    }
  }
  return best_eff > 0 ? best : fb;
}

// bf16 shapes always take the tensor-core path: sm_103 and at most 256 rows
// (buddy_create rejects anything else).
bool gemm_tc_supported(const Ctx& c) {
  if (c.dtype != BUDDY_DTYPE_BF16 || c.maxB > 256 || (c.hd != 64 && c.hd != 128)) return false;
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, c.device);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, c.device);
  return major == 10 && minor == 3 && get_encode() != nullptr;
}

int gemm_tc_prepare(Ctx& c) {
  c.use_tc = c.dtype == BUDDY_DTYPE_BF16;
  if (!c.use_tc) return BUDDY_OK;
  if (!gemm_tc_supported(c)) return BUDDY_ERR_ARG;
  // geometry: 256 weight rows per tile; one M-tile per 128 rows of the batch
  c.tc_bw = kTileN;
  c.tc_mt = c.maxB > 128 ? 2 : 1;
  c.tc_rows_max = std::max(16, (c.maxB + 15) & ~15);
  c.tc_xr = c.tc_mt == 1 ? (uint32_t)c.tc_rows_max * 128u : kXTileMax;
  // One CTA per SM with the full ring.
  const int limit = 227 * 1024 - 2 * 1024;   // room for static shared memory
  c.tc_acc_bufs = c.tc_mt == 2 ? 1 : 2;
  c.tc_tmem_cols = 512;
  for (int v = 0; v < 2; ++v) {
    const uint32_t stage_bytes = (uint32_t)c.tc_bw * 128u + (uint32_t)(v + 1) * c.tc_mt * c.tc_xr;
    c.tc_stages[v] = std::min(kTcMaxStages, (int)((limit - 1024) / stage_bytes));
    c.tc_stage_bytes[v] = stage_bytes;
    c.tc_w_off[v] = (uint32_t)(v + 1) * c.tc_mt * c.tc_xr;
    c.tc_smem[v] = c.tc_stages[v] * stage_bytes + 1024;
  }
  size_t ws = 0;
  int max_tiles = 1;
  for (int w = 0; w < 4; ++w) {
    int N, K, tiles;
    gemm_shape(c, w, &N, &K, &tiles);
    const int kb = (K + kTileK - 1) / kTileK;
    c.tc_splits[w] = choose_splits(tiles, kb, c.num_sms);
    c.tc_tiles[w] = tiles;
    // every unit stages its accumulator rows in the workspace
    ws = std::max(ws, (size_t)tiles * c.tc_splits[w] * c.tc_rows_max * c.tc_bw);
    max_tiles = std::max(max_tiles, tiles);
  }
  // tensor maps: activations (fixed scratch) and per-layer weights
  c.tmaps_host.assign((size_t)c.L * 4 + 6, CUtensorMap{});
  CUtensorMap* X = &c.tmaps_host[(size_t)c.L * 4];
  if (!make_map(&X[0], c.xn, c.maxB, c.d, 16) || !make_map(&X[1], c.attn_out, c.maxB, c.qd, 16) ||
      !make_map(&X[2], c.act, c.maxB, c.F, 16) || !make_map(&X[3], c.xn_lo, c.maxB, c.d, 16) ||
      !make_map(&X[4], c.attn_lo, c.maxB, c.qd, 16) || !make_map(&X[5], c.act_lo, c.maxB, c.F, 16))
    return BUDDY_ERR_CUDA;
  for (int l = 0; l < c.L; ++l) {
    const buddy_layer_weights& w = c.layers[l];
    CUtensorMap* M = &c.tmaps_host[(size_t)l * 4];
    const uint32_t bw = (uint32_t)c.tc_bw;
    if (!make_map(&M[0], w.w_qkv, c.qkvN, c.d, bw) || !make_map(&M[1], w.w_o, c.d, c.qd, bw) ||
        !make_map(&M[2], w.w_gate_up, 2ull * c.F, c.d, bw / 2) || !make_map(&M[3], w.w_down, c.d, c.F, bw))
      return BUDDY_ERR_ARG;
  }
  if (ws > c.gemm_ws_elems) {
    if (c.gemm_ws) cudaFree(c.gemm_ws);
    c.gemm_ws = nullptr;
    if (cudaMalloc(&c.gemm_ws, ws * sizeof(float)) != cudaSuccess) return BUDDY_ERR_CUDA;
    c.gemm_ws_elems = ws;
  }
  if (max_tiles > c.gemm_ctr_n) {
    if (c.gemm_ctr) cudaFree(c.gemm_ctr);
    c.gemm_ctr = nullptr;
    if (cudaMalloc(&c.gemm_ctr, max_tiles * sizeof(int32_t)) != cudaSuccess) return BUDDY_ERR_CUDA;
    c.gemm_ctr_n = max_tiles;
  }
  if (cudaMemset(c.gemm_ctr, 0, c.gemm_ctr_n * sizeof(int32_t)) != cudaSuccess) return BUDDY_ERR_CUDA;
  // Panel mode for up to eight rows: the QKV and gate/up GEMMs normalise their
  // own activations (no RMSNorm kernels, no activation copies).  Stages hold
  // weight tiles only; two panels of the largest K range follow the ring, then
  // 15 KiB for the tail of an M = 128 operand read, then the first unit's
  // RMSNorm gains (staged before the dependency wait).
  c.tc_panel = c.maxB <= 8 && c.d % kTileK == 0;
  if (c.tc_panel) {
    int N, K, tiles;
    gemm_shape(c, 0, &N, &K, &tiles);
    c.tc_panel_kb = (K / kTileK + c.tc_splits[0] - 1) / c.tc_splits[0];
    gemm_shape(c, 2, &N, &K, &tiles);
    c.tc_panel_kb = std::max(c.tc_panel_kb, (K / kTileK + c.tc_splits[2] - 1) / c.tc_splits[2]);
    const int limit = 227 * 1024 - 2 * 1024;
    for (int v = 0; v < 2; ++v) {
      c.tc_panel_bytes[v] = (uint32_t)(v + 1) * (uint32_t)c.tc_panel_kb * 1024u;
      // + the first unit's RMSNorm gains (fp32)
      const int fixed = 1024 + 2 * (int)c.tc_panel_bytes[v] + 15 * 1024 + c.tc_panel_kb * kTileK * 4;
      c.tc_pstages[v] = std::min(kTcMaxStages, (limit - fixed) / (c.tc_bw * 128));
      c.tc_psmem[v] = c.tc_pstages[v] * c.tc_bw * 128 + fixed;
      if (c.tc_pstages[v] < 3) c.tc_panel = false;
    }
  }
  // Above kTcDeferRows rows a tile's partials are too many for the one CTA
  // that would finish it (m x 256 fp32 per split): a fixup kernel spreads
  // them over all SMs.
  c.tc_defer = c.maxB > kTcDeferRows;
  if (c.pf_max > 0) {
    // prefill activations: 128-row boxes (one M-tile per copy)
    if (!make_map(&c.pf_tmaps[0], c.pf_xn, c.pf_max, c.d, 128) ||
        !make_map(&c.pf_tmaps[1], c.pf_attn, c.pf_max, c.qd, 128) ||
        !make_map(&c.pf_tmaps[2], c.pf_act, c.pf_max, c.F, 128) ||
        !make_map(&c.pf_tmaps[3], c.pf_xn_lo, c.pf_max, c.d, 128) ||
        !make_map(&c.pf_tmaps[4], c.pf_attn_lo, c.pf_max, c.qd, 128) ||
        !make_map(&c.pf_tmaps[5], c.pf_act_lo, c.pf_max, c.F, 128))
      return BUDDY_ERR_CUDA;
    const int rc = gemm_pf_prepare(c);
    if (rc != BUDDY_OK) return rc;
  }
  const cudaFuncAttribute A = cudaFuncAttributeMaxDynamicSharedMemorySize;
  const int qs0 = std::max(c.tc_smem[0], c.tc_panel ? c.tc_psmem[0] : 0);
  const int qs1 = std::max(c.tc_smem[1], c.tc_panel ? c.tc_psmem[1] : 0);
  if (cudaFuncSetAttribute(gemm_tc_kernel<EPI_STORE_F32, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_SWIGLU, false>, A, qs0) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_STORE_F32, true>, A, c.tc_smem[1]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID, true>, A, c.tc_smem[1]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_SWIGLU, true>, A, qs1) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_QKV, false>, A, qs0) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_QKV, true>, A, qs1))
    return BUDDY_ERR_CUDA;
  return BUDDY_OK;
}

// Kernel parameters of one GEMM call; *smem = its dynamic shared memory.
static TcParams tc_params(const Ctx& c, const GemmArgs& a, size_t* smem_out) {
  const int which = a.which;
  TcParams p{};
  int N, K, tiles;
  gemm_shape(c, which, &N, &K, &tiles);
  p.N = N;
  p.K = K;
  p.n_tiles = tiles;
  p.kb_total = (K + kTileK - 1) / kTileK;
  p.splits = c.tc_splits[which];
  p.kb_per_split = (p.kb_total + p.splits - 1) / p.splits;
  p.units = tiles * p.splits;
  p.bw = c.tc_bw;
  p.mt = c.tc_mt;
  p.rows_max = c.tc_rows_max;
  const int v = a.split ? 1 : 0;
  p.stages = c.tc_stages[v];
  p.acc_bufs = c.tc_acc_bufs;
  p.stage_bytes = c.tc_stage_bytes[v];
  p.xr = c.tc_xr;
  p.w_off = c.tc_w_off[v];
  p.tmem_cols = c.tc_tmem_cols;
  p.rows = a.sel.rows;
  p.count = a.sel.count;
  p.n = a.sel.n;
  p.out_f32 = a.out_f32;
  p.out_act = (bf16*)a.out_act;
  p.out_act_lo = (bf16*)a.out_act_lo;
  p.resid_src = a.resid_src;
  p.resid_dst = a.resid_dst;
  p.ws = c.gemm_ws;
  p.ctr = c.gemm_ctr;
  p.status = c.status;
  p.bias = a.qkv_bias;
  p.rope_cos = c.rope_cos;
  p.rope_sin = c.rope_sin;
  p.len = a.kv_len;
  p.cache_len = a.cache_len ? a.cache_len : a.kv_len;
  p.seq_off = a.kv_seq_off;
  p.cap = a.kv_cap;
  p.kc = (bf16*)a.kc;
  p.vc = (bf16*)a.vc;
  p.q_out = a.q_out;
  p.pool = a.pool;
  size_t smem = c.tc_smem[v];
  if (a.in_norm_src) {   // panel mode
    p.nsrc = a.in_norm_src;
    p.ngamma = a.in_norm_gamma;
    p.neps = c.cfg.rms_eps;
    p.stages = c.tc_pstages[v];
    p.stage_bytes = (uint32_t)c.tc_bw * 128u;
    p.w_off = 0;
    p.panel_off = (uint32_t)p.stages * p.stage_bytes;
    p.panel_bytes = c.tc_panel_bytes[v];
    p.gstage_off = p.panel_off + 2 * p.panel_bytes + 15 * 1024;
    p.panel_kb = c.tc_panel_kb;
    smem = c.tc_psmem[v];
  }
  p.count_late = a.count_late ? 1 : 0;
  p.defer = c.tc_defer ? 1 : 0;
  p.wait_ns = c.wait_ns;
  p.nq = c.nq;
  p.nkv = c.nkv;
  p.hd = c.hd;
  *smem_out = smem;
  return p;
}

void launch_gemm_tc(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s) {
  const int which = a.which;
  size_t smem = 0;
  const TcParams p = tc_params(c, a, &smem);
  const CUtensorMap& tw = c.tmaps_host[(size_t)a.layer * 4 + which];
  const int xi = which == 0 || which == 2 ? 0 : (which == 1 ? 1 : 2);
  const CUtensorMap& tx = c.tmaps_host[(size_t)c.L * 4 + xi];
  const CUtensorMap& txlo = c.tmaps_host[(size_t)c.L * 4 + 3 + xi];
  const int grid = std::min(p.units, c.num_sms);

  if (a.split) {
    switch (epi) {
      case EPI_QKV:
        launch_k(gemm_tc_kernel<EPI_QKV, true>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      case EPI_STORE_F32:
        launch_k(gemm_tc_kernel<EPI_STORE_F32, true>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      case EPI_RESID:
        launch_k(gemm_tc_kernel<EPI_RESID, true>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      default:
        launch_k(gemm_tc_kernel<EPI_SWIGLU, true>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
    }
  } else {
    switch (epi) {
      case EPI_QKV:
        launch_k(gemm_tc_kernel<EPI_QKV, false>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      case EPI_STORE_F32:
        launch_k(gemm_tc_kernel<EPI_STORE_F32, false>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      case EPI_RESID:
        launch_k(gemm_tc_kernel<EPI_RESID, false>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
        break;
      default:
        launch_k(gemm_tc_kernel<EPI_SWIGLU, false>, grid, kTcThreads, smem, s, c.pdl, tw, tx, txlo, p);
    }
  }
}

void launch_gemm_fix(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s) {
  size_t smem = 0;
  const TcParams p = tc_params(c, a, &smem);
  const int fgrid = c.num_sms * (2048 / kTcFixThreads);
  if (a.split) {
    switch (epi) {
      case EPI_QKV: launch_k(gemm_fix_kernel<EPI_QKV, true>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      case EPI_STORE_F32: launch_k(gemm_fix_kernel<EPI_STORE_F32, true>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      case EPI_RESID: launch_k(gemm_fix_kernel<EPI_RESID, true>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      default: launch_k(gemm_fix_kernel<EPI_SWIGLU, true>, fgrid, kTcFixThreads, 0, s, c.pdl, p);
    }
  } else {
    switch (epi) {
      case EPI_QKV: launch_k(gemm_fix_kernel<EPI_QKV, false>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      case EPI_STORE_F32: launch_k(gemm_fix_kernel<EPI_STORE_F32, false>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      case EPI_RESID: launch_k(gemm_fix_kernel<EPI_RESID, false>, fgrid, kTcFixThreads, 0, s, c.pdl, p); break;
      default: launch_k(gemm_fix_kernel<EPI_SWIGLU, false>, fgrid, kTcFixThreads, 0, s, c.pdl, p);
    }
  }
}


}  // namespace buddy

// Tensor-core GEMM for the bf16 decode projections on sm_103a.
//
//   C[j][n] = sum_k X[j][k] * W[n][k]      (j < m active rows, n < N features)
//
// Decode GEMMs are skinny (m = 1..256) and bound by streaming W from HBM, so
// the operands are swapped: a 128-row weight tile is the MMA's M side and the
// m active rows (padded to a multiple of 16) are its N side.  Both operands are
// K-major bf16 tiles of 64 columns staged in shared memory by TMA with 128-byte
// swizzle; tcgen05.mma accumulates fp32 in TMEM.  Persistent CTAs (one per SM)
// walk work units (weight tile, K split); warp 0 issues TMA loads into a ring
// of stages, warp 1 issues the MMAs, warps 2-5 drain TMEM (double-buffered
// accumulators) and run the epilogue.  A tile split over K is finished by the
// last CTA to arrive, which sums the partials in split order (deterministic).
//
// Epilogues: fp32 store; residual add into the (row-gathered) hidden state;
// SwiGLU, where a tile holds 64 gate rows and the matching 64 up rows.
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
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ volatile int consumed;
  __shared__ int last_flag;
  __shared__ float xch[128 * 17];

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
        uint8_t* a = smem + (size_t)npre * p.stage_bytes;
        ptx::mbar_expect_tx(&full_bar[npre], kTileABytes);
        if (EPI == EPI_SWIGLU) {
          ptx::tma_load_2d_hint(a, &tw, &full_bar[npre], kb * kTileK, tile * 64, pol);
          ptx::tma_load_2d_hint(a + kTileABytes / 2, &tw, &full_bar[npre], kb * kTileK, p.N + tile * 64, pol);
        } else {
          ptx::tma_load_2d_hint(a, &tw, &full_bar[npre], kb * kTileK, tile * 128, pol);
        }
      }
    }
  }
  pdl_wait();
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
  const int BN = max(16, (m + 15) & ~15);
  const uint32_t x_bytes = (SPLIT ? 2u : 1u) * (uint32_t)BN * 128u;
  const uint32_t lo_off = kTileABytes + (uint32_t)p.bn_max * 128u;   // B_lo tile offset in a stage

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
          uint8_t* a = smem + (size_t)stage * p.stage_bytes;
          uint8_t* b = a + kTileABytes;
          if (issued < npre) {
            // weight tile already in flight: add the activation tile
            ptx::mbar_arrive_expect_tx(&full_bar[stage], x_bytes);
          } else {
            if (!ptx::mbar_wait_bounded(&empty_bar[stage], ph ^ 1u, kWaitLimitNs, &abort_flag)) {
              ok = false;
              break;
            }
            ptx::mbar_arrive_expect_tx(&full_bar[stage], kTileABytes + x_bytes);
            if (EPI == EPI_SWIGLU) {
              ptx::tma_load_2d_hint(a, &tw, &full_bar[stage], kb * kTileK, tile * 64, pol);
              ptx::tma_load_2d_hint(a + kTileABytes / 2, &tw, &full_bar[stage], kb * kTileK, p.N + tile * 64,
                                    pol);
            } else {
              ptx::tma_load_2d_hint(a, &tw, &full_bar[stage], kb * kTileK, tile * 128, pol);
            }
          }
          for (int r = 0; r < BN / 16; ++r) {
            ptx::tma_load_2d(b + r * 2048, &tx, &full_bar[stage], kb * kTileK, r * 16);
            if (SPLIT) ptx::tma_load_2d(a + lo_off + r * 2048, &txlo, &full_bar[stage], kb * kTileK, r * 16);
          }
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
      const uint32_t idesc = ptx::idesc_bf16_m128((uint32_t)BN);
      int stage = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      int n_consumed = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
        const int split = u / p.n_tiles;
        const int kb0 = split * p.kb_per_split, kb1 = min(p.kb_total, kb0 + p.kb_per_split);
        if (!ptx::mbar_wait_bounded(&tempty_bar[acc], acc_ph ^ 1u, kWaitLimitNs, &abort_flag)) break;
        ptx::tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(acc * p.bn_max);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!ptx::mbar_wait_bounded(&full_bar[stage], ph, kWaitLimitNs, &abort_flag)) {
            ok = false;
            break;
          }
          consumed = ++n_consumed;
          ptx::tc_fence_after();
          const uint8_t* a = smem + (size_t)stage * p.stage_bytes;
          const uint64_t da = ptx::smem_desc_sw128(a);
          const uint64_t db = ptx::smem_desc_sw128(a + kTileABytes);
#pragma unroll
          for (int k = 0; k < kTileK / 16; ++k) {
            ptx::mma_bf16(d, da + 2ull * k, db + 2ull * k, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
            if (SPLIT) {
              const uint64_t dl = ptx::smem_desc_sw128(a + lo_off);
              ptx::mma_bf16(d, da + 2ull * k, dl + 2ull * k, idesc, 1u);
            }
          }
          ptx::mma_commit(&empty_bar[stage]);
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        ptx::mma_commit(&tfull_bar[acc]);
        acc ^= 1;
        if (acc == 0) acc_ph ^= 1u;
      }
      // all issued MMAs complete before TMEM is released
      ptx::mma_commit(&done_bar);
      volatile int dummy = 0;
      ptx::mbar_wait_bounded(&done_bar, 0, kWaitLimitNs, &dummy);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- epilogue
    const int lane_base = (warp & 3) * 32;
    const int row = lane_base + lane;
    int acc = 0;
    uint32_t acc_ph = 0;
    for (int u = blockIdx.x; u < p.units; u += gridDim.x) {
      const int tile = u % p.n_tiles, split = u / p.n_tiles;
      const bool ok = ptx::mbar_wait_bounded(&tfull_bar[acc], acc_ph, kWaitLimitNs, &abort_flag);
      if (epi_bar_any(!ok)) break;
      ptx::tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)lane_base << 16) + (uint32_t)(acc * p.bn_max);
      float v[16];
      if (p.splits == 1) {
        for (int c0 = 0; c0 < BN; c0 += 16) {
          ptx::tmem_ld16(taddr + c0, v);
          apply_epilogue<EPI, SPLIT>(p, tile, row, c0, m, v, xch);
        }
        ptx::tc_fence_before();
        if (lane == 0) ptx::mbar_arrive(&tempty_bar[acc]);
      } else {
        float* slot = p.ws + (size_t)u * p.bn_max * 128;
        for (int c0 = 0; c0 < BN; c0 += 16) {
          ptx::tmem_ld16(taddr + c0, v);
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (c0 + i < m) __stcg(slot + (size_t)(c0 + i) * 128 + row, v[i]);
        }
        ptx::tc_fence_before();
        if (lane == 0) ptx::mbar_arrive(&tempty_bar[acc]);
        epi_bar();
        if (threadIdx.x == 64) {
          __threadfence();
          const int old = atomicAdd(&p.ctr[tile], 1);
          last_flag = (old == p.splits - 1);
          if (last_flag) p.ctr[tile] = 0;
          __threadfence();
        }
        epi_bar();
        if (last_flag) {
          __threadfence();
          for (int c0 = 0; c0 < BN; c0 += 16) {
            const int nc = min(16, m - c0);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = 0.f;
            // four splits' loads in flight per round, summed in split order
            for (int s = 0; s < p.splits; s += 4) {
              float t[4][16];
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float* sl = p.ws + (size_t)((s + q) * p.n_tiles + tile) * p.bn_max * 128 + row;
#pragma unroll
                for (int i = 0; i < 16; ++i)
                  t[q][i] = (s + q < p.splits && i < nc) ? __ldcg(sl + (size_t)(c0 + i) * 128) : 0.f;
              }
#pragma unroll
              for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int i = 0; i < 16; ++i) v[i] += t[q][i];
            }
            apply_epilogue<EPI, SPLIT>(p, tile, row, c0, m, v, xch);
          }
        }
        epi_bar();
      }
      acc ^= 1;
      if (acc == 0) acc_ph ^= 1u;
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (threadIdx.x == 0 && abort_flag) atomicOr(p.status, BUDDY_DEV_TIMEOUT);
  if (warp == 1) ptx::tmem_dealloc(tmem_base, p.tmem_cols);
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

// Split-K factor: the smallest one whose last wave of persistent CTAs is at
// least 80% busy (every split >= 4 K-blocks); fewer splits mean fewer
// per-unit epilogues and partial sums.  Falls back to the best efficiency.
static int choose_splits(int tiles, int kb, int sms) {
  int best = 1;
  double best_eff = -1.0;
  for (int s = 1; s <= 32; ++s) {
    const int kps = (kb + s - 1) / s;
    if (s > 1 && (kps < 4 || (s - 1) * kps >= kb)) continue;
    const int units = tiles * s;
    const int waves = (units + sms - 1) / sms;
    const double eff = (double)units / (double)(waves * sms);
    if (eff >= 0.8) return s;
    if (eff > best_eff + 0.02) {
      best_eff = eff;
      best = s;
    }
  }
  return best;
}

bool gemm_tc_supported(const Ctx& c) {
  if (c.dtype != BUDDY_DTYPE_BF16 || c.maxB > 256) return false;
  const char* env = getenv("BUDDY_GEMM");
  if (env && env[0] == 's') return false;   // "simt": CUDA-core kernel for every GEMM
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, c.device);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, c.device);
  return major == 10 && minor == 3 && get_encode() != nullptr;
}

int gemm_tc_prepare(Ctx& c) {
  c.use_tc = gemm_tc_supported(c);
  c.use_lk = false;
  if (!c.use_tc) return BUDDY_OK;
  c.tc_bn_max = std::max(16, (c.maxB + 15) & ~15);
  const int smem_limit = 227 * 1024 - 12 * 1024;  // leave room for static shared memory (~9.5 KiB)
  for (int v = 0; v < 2; ++v) {
    const uint32_t stage_bytes = kTileABytes + (uint32_t)(v + 1) * (uint32_t)c.tc_bn_max * 128u;
    c.tc_stages[v] = std::min(kTcMaxStages, (int)((smem_limit - 1024) / stage_bytes));
    c.tc_stage_bytes[v] = stage_bytes;
    c.tc_smem[v] = c.tc_stages[v] * stage_bytes + 1024;
  }
  uint32_t cols = 32;
  while (cols < 2u * (uint32_t)c.tc_bn_max) cols <<= 1;
  c.tc_tmem_cols = cols;
  size_t ws = 0;
  int max_tiles = 1;
  for (int w = 0; w < 4; ++w) {
    int N, K, tiles;
    gemm_shape(c, w, &N, &K, &tiles);
    const int kb = (K + kTileK - 1) / kTileK;
    c.tc_splits[w] = choose_splits(tiles, kb, c.num_sms);
    c.tc_tiles[w] = tiles;
    if (c.tc_splits[w] > 1) ws = std::max(ws, (size_t)tiles * c.tc_splits[w] * c.tc_bn_max * 128);
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
    if (!make_map(&M[0], w.w_qkv, c.qkvN, c.d, 128) || !make_map(&M[1], w.w_o, c.d, c.qd, 128) ||
        !make_map(&M[2], w.w_gate_up, 2ull * c.F, c.d, 64) || !make_map(&M[3], w.w_down, c.d, c.F, 128))
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
  const char* lk_env = getenv("BUDDY_LAYER_KERNEL");
  c.use_lk = layer_kernel_supported(c) && lk_env && lk_env[0] == '1';   // opt-in
  if (c.use_lk && !c.lk_bar) {
    if (cudaMalloc(&c.lk_bar, 2 * sizeof(unsigned)) != cudaSuccess) return BUDDY_ERR_CUDA;
    if (cudaMemset(c.lk_bar, 0, 2 * sizeof(unsigned)) != cudaSuccess) return BUDDY_ERR_CUDA;
  }
  const cudaFuncAttribute A = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if (cudaFuncSetAttribute(gemm_tc_kernel<EPI_STORE_F32, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_SWIGLU, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_STORE_F32, true>, A, c.tc_smem[1]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID, true>, A, c.tc_smem[1]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_SWIGLU, true>, A, c.tc_smem[1]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_QKV, false>, A, c.tc_smem[0]) ||
      cudaFuncSetAttribute(gemm_tc_kernel<EPI_QKV, true>, A, c.tc_smem[1]))
    return BUDDY_ERR_CUDA;
  return BUDDY_OK;
}

void launch_gemm_tc(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s) {
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
  p.bn_max = c.tc_bn_max;
  const int v = a.split ? 1 : 0;
  p.stages = c.tc_stages[v];
  p.stage_bytes = c.tc_stage_bytes[v];
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
  p.seq_off = a.kv_seq_off;
  p.cap = a.kv_cap;
  p.kc = (bf16*)a.kc;
  p.vc = (bf16*)a.vc;
  p.q_out = a.q_out;
  p.pool = a.pool;
  p.nq = c.nq;
  p.nkv = c.nkv;
  p.hd = c.hd;
  const CUtensorMap& tw = c.tmaps_host[(size_t)a.layer * 4 + which];
  const int xi = which == 0 || which == 2 ? 0 : (which == 1 ? 1 : 2);
  const CUtensorMap& tx = c.tmaps_host[(size_t)c.L * 4 + xi];
  const CUtensorMap& txlo = c.tmaps_host[(size_t)c.L * 4 + 3 + xi];
  const int grid = std::min(p.units, c.num_sms);
  const size_t smem = c.tc_smem[v];
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

}  // namespace buddy

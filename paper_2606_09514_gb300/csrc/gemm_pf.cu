// Tensor-core GEMM for the prefill projections on sm_103a.
//
//   C[j][n] = sum_k X[j][k] * W[n][k]      (j < m prompt-token rows, n < N features)
//
// A prefill block runs its projections on every token of the prompts that
// selected it, thousands of rows: the GEMM is bound by the tensor pipe, not
// by the weight stream.  A work unit is one 128-row M-tile of X times one
// 256-row weight tile over the whole K (no split); persistent CTAs (one per
// SM) walk the units M-tile by M-tile, so the CTAs running at any time share
// a few activation tiles and stream the weight tiles from L2.
//
// Warp 0 issues the TMA loads of a ring of stages ([X 128 x 64][X remainder
// 128 x 64 with SPLIT][W 256 x 64], 128-byte swizzle); warp 1 issues
// tcgen05.mma M = 128, N = 256, K = 16 into one of two TMEM accumulators
// (512 columns); warps 2-5 drain the other accumulator and apply the
// epilogue, each thread one row of the tile.  Every wait is bounded.
//
// Epilogues: residual add scattered to the token rows; SwiGLU (a tile holds
// 128 gate rows and the matching 128 up rows); QKV (bias, rotate-half RoPE at
// the token's position, q out in fp32, K/V stored in the layer's cache at the
// token's cache position).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "common.cuh"
#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace buddy {

constexpr int kPfThreads = 192;
constexpr int kPfMaxStages = 8;
constexpr uint32_t kPfABytes = 128u * 128u;   // one 128-row x 64-column bf16 tile
constexpr uint32_t kPfWBytes = 256u * 128u;   // one 256-row weight tile

struct PfParams {
  int N, K, m;
  int n_tiles, m_tiles, kb_total, units;
  int stages;
  uint32_t stage_bytes, w_off;
  // epilogue
  const int32_t* rows;     // compact row j -> token row (residual, QKV); nullptr = identity
  const float* resid_src;
  float* resid_dst;
  bf16* out_act;
  bf16* out_act_lo;
  float* q_out;            // [m, nq * hd] compact
  const float* bias;
  const float* rope_cos;
  const float* rope_sin;
  const int32_t* tok_seq;  // token row -> sequence
  const int32_t* tok_pos;  // token row -> RoPE position
  const int32_t* len;      // sequence -> tokens before this prefill
  const int32_t* cache_len;  // sequence -> the layer's positions before this prefill
  const int64_t* seq_off;
  const int32_t* cap;
  bf16* kc;
  bf16* vc;
  int nq, nkv, hd;
  int32_t* status;
  uint64_t wait_ns;        // limit of each pipeline wait (the drain waits keep kWaitLimitNs)
};

template <int EPI>
__device__ __forceinline__ void pf_load_w(uint8_t* st, const CUtensorMap* tw, uint64_t* bar, const PfParams& p,
                                          int tile, int kb) {
  if (EPI == EPI_SWIGLU) {   // gate rows f0.., then the matching up rows N + f0..
    ptx::tma_load_2d(st, tw, bar, kb * kTileK, tile * 128);
    ptx::tma_load_2d(st + 128 * 128, tw, bar, kb * kTileK, p.N + tile * 128);
  } else {
    ptx::tma_load_2d(st, tw, bar, kb * kTileK, tile * 256);
  }
}

__device__ __forceinline__ void st_bf16x8(bf16* dst, const float* v) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
    w[i] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[2 * i])) |
           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[2 * i + 1])) << 16);
  *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

// QKV epilogue of row j: the tile's 256 columns are 256 / HD whole heads;
// bias, rotate-half RoPE at the token's position (pairs e, e + HD/2), q out in
// fp32, K/V stored (bf16) at the token's position in the layer's cache.
template <int HD>
__device__ __forceinline__ void pf_qkv(const PfParams& p, int j, int nt, uint32_t ta) {
  constexpr int half = HD / 2;
  const bool live = j < p.m;
  int seq = 0, pos = 0, cpos = 0;
  if (live) {
    const int row = p.rows ? p.rows[j] : j;
    seq = p.tok_seq[row];
    pos = p.tok_pos[row];
    cpos = p.cache_len[seq] + (pos - p.len[seq]);
  }
#pragma unroll 1
  for (int cb = 0; cb < 256; cb += HD) {
    float x[HD];
    ptx::tmem_ld64(ta + cb, x);
    if (HD == 128) ptx::tmem_ld64(ta + cb + 64, x + 64);
    const int n0 = nt * 256 + cb;   // first feature of this head
    if (!live || n0 >= p.N) continue;
    const int head = n0 / HD;
    if (p.bias) {
#pragma unroll
      for (int e = 0; e < HD; ++e) x[e] += p.bias[n0 + e];
    }
    if (head < p.nq + p.nkv) {
      const float* co = p.rope_cos + (size_t)pos * half;
      const float* si = p.rope_sin + (size_t)pos * half;
#pragma unroll
      for (int e = 0; e < half; ++e) {
        const float a = x[e], b = x[e + half];
        x[e] = a * co[e] - b * si[e];
        x[e + half] = b * co[e] + a * si[e];
      }
      if (head < p.nq) {
        float4* q = reinterpret_cast<float4*>(p.q_out + (size_t)j * p.nq * HD + (size_t)head * HD);
#pragma unroll
        for (int e = 0; e < HD; e += 4) q[e >> 2] = make_float4(x[e], x[e + 1], x[e + 2], x[e + 3]);
      } else {
        bf16* k = p.kc + kv_offset(p.seq_off, p.cap, seq, p.nkv, HD, head - p.nq, cpos);
#pragma unroll
        for (int e = 0; e < HD; e += 8) st_bf16x8(k + e, x + e);
      }
    } else {
      bf16* v = p.vc + kv_offset(p.seq_off, p.cap, seq, p.nkv, HD, head - p.nq - p.nkv, cpos);
#pragma unroll
      for (int e = 0; e < HD; e += 8) st_bf16x8(v + e, x + e);
    }
  }
}

// Epilogue of row j (lane of this warp's TMEM quarter) of unit tile nt.  All
// lanes run the TMEM loads (warp-collective); only rows j < m store.
template <int EPI, bool SPLIT>
__device__ __forceinline__ void pf_epilogue(const PfParams& p, int j, int nt, uint32_t ta) {
  const bool live = j < p.m;
  if (EPI == EPI_RESID) {
    const int row = live ? (p.rows ? p.rows[j] : j) : 0;
    for (int c0 = 0; c0 < 256; c0 += 64) {
      float v[64];
      ptx::tmem_ld64(ta + c0, v);
      const int n0 = nt * 256 + c0;
      if (!live || n0 >= p.N) continue;   // N is a multiple of 64
      const float4* src = reinterpret_cast<const float4*>(p.resid_src + (size_t)row * p.N + n0);
      float4* dst = reinterpret_cast<float4*>(p.resid_dst + (size_t)row * p.N + n0);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float4 s = src[i];
        dst[i] = make_float4(s.x + v[4 * i], s.y + v[4 * i + 1], s.z + v[4 * i + 2], s.w + v[4 * i + 3]);
      }
    }
  } else if (EPI == EPI_SWIGLU) {
    for (int h = 0; h < 128; h += 64) {
      float g[64], u[64];
      ptx::tmem_ld64(ta + h, g);
      ptx::tmem_ld64(ta + 128 + h, u);
      if (!live) continue;
      const int f0 = nt * 128 + h;
#pragma unroll
      for (int i = 0; i < 64; i += 8) {
        if (f0 + i >= p.N) break;   // N is a multiple of 8
        float a[8], lo[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          a[e] = silu_f(g[i + e]) * u[i + e];
          lo[e] = a[e] - __bfloat162float(__float2bfloat16_rn(a[e]));
        }
        st_bf16x8(p.out_act + (size_t)j * p.N + f0 + i, a);
        if (SPLIT) st_bf16x8(p.out_act_lo + (size_t)j * p.N + f0 + i, lo);
      }
    }
  } else if (p.hd == 128) {
    pf_qkv<128>(p, j, nt, ta);
  } else {
    pf_qkv<64>(p, j, nt, ta);
  }
}

template <int EPI, bool SPLIT>
__global__ void __launch_bounds__(kPfThreads, 1)
    gemm_pf_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tx,
                   const __grid_constant__ CUtensorMap txlo, const PfParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kPfMaxStages], empty_bar[kPfMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ volatile int consumed;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  if (call_aborted(p.status)) return;

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
    ptx::tmem_alloc(&tmem_slot, 512);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA
    if (lane == 0) {
      const uint32_t bytes = (SPLIT ? 2u : 1u) * kPfABytes + kPfWBytes;
      int stage = 0;
      uint32_t ph = 0;
      int issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
        const int mt = u / p.n_tiles, nt = u - mt * p.n_tiles;
        for (int kb = 0; kb < p.kb_total; ++kb) {
          if (!ptx::mbar_wait_bounded(&empty_bar[stage], ph ^ 1u, p.wait_ns, &abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + (size_t)stage * p.stage_bytes;
          ptx::mbar_arrive_expect_tx(&full_bar[stage], bytes);
          ptx::tma_load_2d(st, &tx, &full_bar[stage], kb * kTileK, mt * 128);
          if (SPLIT) ptx::tma_load_2d(st + kPfABytes, &txlo, &full_bar[stage], kb * kTileK, mt * 128);
          pf_load_w<EPI>(st + p.w_off, &tw, &full_bar[stage], p, nt, kb);
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
      const uint32_t idesc = ptx::idesc_bf16(128u, 256u);
      int stage = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      int n_consumed = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
        if (!ptx::mbar_wait_bounded(&tempty_bar[acc], acc_ph ^ 1u, p.wait_ns, &abort_flag)) break;
        ptx::tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)acc * 256u;
        for (int kb = 0; kb < p.kb_total; ++kb) {
          if (!ptx::mbar_wait_bounded(&full_bar[stage], ph, p.wait_ns, &abort_flag)) {
            ok = false;
            break;
          }
          consumed = ++n_consumed;
          ptx::tc_fence_after();
          const uint8_t* st = smem + (size_t)stage * p.stage_bytes;
          const uint64_t da = ptx::smem_desc_sw128(st);
          const uint64_t dl = ptx::smem_desc_sw128(st + kPfABytes);
          const uint64_t dw = ptx::smem_desc_sw128(st + p.w_off);
#pragma unroll
          for (int k = 0; k < kTileK / 16; ++k) {
            ptx::mma_bf16(d, da + 2ull * k, dw + 2ull * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
            if (SPLIT) ptx::mma_bf16(d, dl + 2ull * k, dw + 2ull * k, idesc, 1u);
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
    const int q = warp & 3;   // TMEM lane quarter this warp may access
    int acc = 0;
    uint32_t acc_ph = 0;
    for (int u = blockIdx.x; u < p.units; u += gridDim.x) {
      const bool ok = ptx::mbar_wait_bounded(&tfull_bar[acc], acc_ph, p.wait_ns, &abort_flag);
      if (epi_bar_any(!ok)) break;
      ptx::tc_fence_after();
      const int mt = u / p.n_tiles, nt = u - mt * p.n_tiles;
      const int j = mt * 128 + q * 32 + lane;
      const uint32_t ta = tmem_base + (uint32_t)acc * 256u + ((uint32_t)(q * 32) << 16);
      pf_epilogue<EPI, SPLIT>(p, j, nt, ta);
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&tempty_bar[acc]);
      acc ^= 1;
      if (acc == 0) acc_ph ^= 1u;
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (threadIdx.x == 0 && abort_flag) atomicOr(p.status, BUDDY_DEV_TIMEOUT);
  if (warp == 1) ptx::tmem_dealloc(tmem_base, 512);
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
int gemm_pf_prepare(Ctx& c) {
  const int limit = 227 * 1024 - 2 * 1024;
  for (int v = 0; v < 2; ++v) {
    const uint32_t sb = (v ? 2u : 1u) * kPfABytes + kPfWBytes;
    c.pf_stages[v] = std::min(kPfMaxStages, (int)((limit - 1024) / sb));
    c.pf_smem[v] = (int)(c.pf_stages[v] * sb) + 1024;
  }
  const cudaFuncAttribute A = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if (cudaFuncSetAttribute(gemm_pf_kernel<EPI_QKV, false>, A, c.pf_smem[0]) ||
      cudaFuncSetAttribute(gemm_pf_kernel<EPI_RESID, false>, A, c.pf_smem[0]) ||
      cudaFuncSetAttribute(gemm_pf_kernel<EPI_SWIGLU, false>, A, c.pf_smem[0]) ||
      cudaFuncSetAttribute(gemm_pf_kernel<EPI_QKV, true>, A, c.pf_smem[1]) ||
      cudaFuncSetAttribute(gemm_pf_kernel<EPI_RESID, true>, A, c.pf_smem[1]) ||
      cudaFuncSetAttribute(gemm_pf_kernel<EPI_SWIGLU, true>, A, c.pf_smem[1]))
    return BUDDY_ERR_CUDA;
  return BUDDY_OK;
}

// One prefill projection: `which` names the weight (0 qkv, 1 o, 2 gate_up,
// 3 down) of `layer`; `xi` the prefill activation map (0 normalised input,
// 1 attention output, 2 SwiGLU output); m rows.
void launch_gemm_pf(const Ctx& c, int epi, bool split, int layer, int which, int xi, int m, const PfEpi& e,
                    cudaStream_t s) {
  PfParams p{};
  int N, K, tiles;
  gemm_shape(c, which, &N, &K, &tiles);
  p.N = N;
  p.K = K;
  p.m = m;
  p.n_tiles = tiles;
  p.m_tiles = (m + 127) / 128;
  p.kb_total = (K + kTileK - 1) / kTileK;
  p.units = p.n_tiles * p.m_tiles;
  const int v = split ? 1 : 0;
  p.stages = c.pf_stages[v];
  p.stage_bytes = (split ? 2u : 1u) * kPfABytes + kPfWBytes;
  p.w_off = (split ? 2u : 1u) * kPfABytes;
  p.rows = e.rows;
  p.resid_src = e.resid_src;
  p.resid_dst = e.resid_dst;
  p.out_act = (bf16*)e.out_act;
  p.out_act_lo = (bf16*)e.out_act_lo;
  p.q_out = e.q_out;
  p.bias = e.bias;
  p.rope_cos = c.rope_cos;
  p.rope_sin = c.rope_sin;
  p.tok_seq = e.tok_seq;
  p.tok_pos = e.tok_pos;
  p.len = e.len;
  p.cache_len = e.cache_len;
  p.seq_off = e.seq_off;
  p.cap = e.cap;
  p.kc = (bf16*)e.kc;
  p.vc = (bf16*)e.vc;
  p.nq = c.nq;
  p.nkv = c.nkv;
  p.hd = c.hd;
  p.status = c.status;
  p.wait_ns = c.wait_ns;
  const CUtensorMap& tw = c.tmaps_host[(size_t)layer * 4 + which];
  const CUtensorMap& tx = c.pf_tmaps[xi];
  const CUtensorMap& txlo = c.pf_tmaps[3 + xi];
  const int grid = std::min(p.units, c.num_sms);
  const size_t smem = c.pf_smem[v];
  if (split) {
    switch (epi) {
      case EPI_QKV: launch_k(gemm_pf_kernel<EPI_QKV, true>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p); break;
      case EPI_RESID: launch_k(gemm_pf_kernel<EPI_RESID, true>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p); break;
      default: launch_k(gemm_pf_kernel<EPI_SWIGLU, true>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p);
    }
  } else {
    switch (epi) {
      case EPI_QKV: launch_k(gemm_pf_kernel<EPI_QKV, false>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p); break;
      case EPI_RESID: launch_k(gemm_pf_kernel<EPI_RESID, false>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p); break;
      default: launch_k(gemm_pf_kernel<EPI_SWIGLU, false>, grid, kPfThreads, smem, s, false, tw, tx, txlo, p);
    }
  }
}

}  // namespace buddy

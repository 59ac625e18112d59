// Building blocks of the tensor-core decode GEMM (gemm_tc.cu).
//
//   C[j][n] = sum_k X[j][k] * W[n][k]      (j < m active rows, n < N features)
//
// Orientation.  A tcgen05.mma instruction (K = 16) takes about 150 cycles
// whatever its M and N, so a decode GEMM, bound by streaming W, must move as
// many weight bytes per instruction as it can.  The active rows are therefore
// the MMA's M side (one or two 128-row M-tiles; rows past m are never read
// back) and a tile of bw = 256 weight rows is its N side: 8 KiB of weights per
// instruction.  (With the weights as M and the rows as N, an instruction moves
// 4 KiB and the instruction rate caps an SM's weight stream near 5 TB/s for
// the whole GPU.)
//
// A stage of the shared-memory ring holds, for one 64-column K block, the
// activation region of each M-tile (then, for the first layer, the regions of
// the bf16 remainder terms) followed by the weight tile [bw rows][128 B], all
// in the 128-byte-swizzled K-major layout.  Only round16(m) activation rows are
// loaded; an M-tile operand always spans 128 rows, so its unused rows read the
// bytes that follow within the stage (their results are discarded).
//
// The accumulator of a unit (tile, K split) is mt x 256 fp32 TMEM columns.
// The ring fills shared memory and, with one M-tile, two accumulators let the
// MMAs of the next unit overlap the epilogue.
//
// Panel mode (up to 8 rows): the ring holds weight tiles only and the
// activations of the QKV and gate/up GEMMs are the RMSNorm of the fp32
// residual rows, computed by the epilogue warps into a shared-memory panel.
//
// Split-K: every unit stages its accumulator rows in a workspace slot; up to
// 8 rows the last split of a tile to arrive sums the slots in split order
// and applies the epilogue, above 8 rows gemm_fix_kernel does so over all
// SMs (tc_ws_idx gives the slot layout).
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace buddy {

constexpr int kTcThreads = 192;
constexpr int kTcMaxStages = 16;
constexpr int kTileK = 64;                       // K columns per stage (128 B of bf16)
constexpr uint32_t kXTileMax = 128 * 128;        // bytes one M-tile operand spans
constexpr int kTileN = 256;                      // weight rows per tile (MMA N)
constexpr uint64_t kWaitLimitNs = 4000000000ull; // 4 s
constexpr int kTcFixThreads = 256;                // deferred-fixup kernel
constexpr int kTcDeferRows = 8;                   // larger batches defer the split-K fixup

struct TcParams {
  int N, K;
  int n_tiles, splits, kb_total, kb_per_split, units;
  int bw, mt;              // weight rows per tile, M-tiles
  uint32_t w_off;          // byte offset of the weight tile in a stage
  int rows_max;            // rows of a workspace slot (round16 of the batch bound)
  int stages, acc_bufs;
  uint32_t stage_bytes, xr, tmem_cols;   // xr: bytes of one M-tile's activation region
  const int32_t* rows;
  const int32_t* count;
  int n;
  float* out_f32;
  bf16* out_act;
  bf16* out_act_lo;       // SPLIT: bf16 remainder of the SwiGLU output
  const float* resid_src;
  float* resid_dst;
  float* ws;
  int32_t* ctr;
  int32_t* status;
  // EPI_QKV: bias, rotate-half RoPE at position len[seq], q out (fp32), K/V
  // appended to the layer's cache, pooled first-layer V
  const float* bias;
  const float* rope_cos;
  const float* rope_sin;
  const int32_t* len;        // RoPE position of each sequence's token
  const int32_t* cache_len;  // cache position of its new entry (len, or the layer's length)
  const int64_t* seq_off;
  const int32_t* cap;
  bf16* kc;
  bf16* vc;
  float* q_out;
  float* pool;
  int nq, nkv, hd;
  // Panel mode (at most 8 rows, K a multiple of 64): the activations are the
  // RMSNorm of the fp32 rows nsrc[rows[j]] (width K), x = bf16(h * rsqrt(
  // mean(h^2) + neps) * ngamma) (+ remainder), computed by the epilogue warps
  // into a shared-memory panel holding the unit's K range (two panels, for the
  // current unit and the next); the ring stages hold weight tiles only.
  const float* nsrc;
  const float* ngamma;
  float neps;
  int count_late;         // the preceding kernel wrote *count: read it after the wait
  uint32_t panel_off;     // byte offset of panel 0 in dynamic shared memory
  uint32_t panel_bytes;   // bytes of one panel (hi, then lo for SPLIT)
  int panel_kb;           // K blocks one panel holds (hi part)
  uint32_t gstage_off;    // byte offset of the first unit's RMSNorm gains (fp32, panel_kb x 64)
  // Deferred fixup: units only stage their partials; a second kernel
  // (gemm_fix_kernel) sums the splits and applies the epilogue on every SM.
  int defer;
  uint64_t wait_ns;       // limit of each pipeline wait (the drain waits keep kWaitLimitNs)
};

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
__device__ __forceinline__ bool epi_bar_any(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n barrier.cta.red.or.pred q, 1, 128, p;\n"
      " selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ int round16(int x) { return (x + 15) & ~15; }

// ---------------------------------------------------------------------------
// Loads of one stage.  The caller has set the barrier's expected bytes.
// ---------------------------------------------------------------------------
// Weight tile `tile` at K block kb.  SwiGLU: the first bw/2 rows are gate rows
// f0.., the next bw/2 the matching up rows N + f0.. (N = F).
template <int EPI>
__device__ __forceinline__ void tc_load_w(uint8_t* stage, const CUtensorMap* tw, uint64_t* bar, const TcParams& p,
                                          int tile, int kb, uint64_t pol) {
  uint8_t* st = stage + p.w_off;
  if (EPI == EPI_SWIGLU) {
    const int h = p.bw >> 1;
    ptx::tma_load_2d_hint(st, tw, bar, kb * kTileK, tile * h, pol);
    ptx::tma_load_2d_hint(st + h * 128, tw, bar, kb * kTileK, p.N + tile * h, pol);
  } else {
    ptx::tma_load_2d_hint(st, tw, bar, kb * kTileK, tile * p.bw, pol);
  }
}

__device__ __forceinline__ uint32_t tc_x_bytes(int m, bool split) {
  return (split ? 2u : 1u) * (uint32_t)round16(m) * 128u;
}

// Activation rows 0..round16(m)-1 at K block kb, 16 rows per copy.
template <bool SPLIT>
__device__ __forceinline__ void tc_load_x(uint8_t* st, const CUtensorMap* tx, const CUtensorMap* txlo, uint64_t* bar,
                                          const TcParams& p, int m, int kb) {
  uint8_t* x0 = st;
  uint8_t* l0 = x0 + p.mt * p.xr;
  for (int r0 = 0; r0 < m; r0 += 16) {
    const uint32_t off = (uint32_t)(r0 >> 7) * p.xr + (uint32_t)(r0 & 127) * 128u;
    ptx::tma_load_2d(x0 + off, tx, bar, kb * kTileK, r0);
    if (SPLIT) ptx::tma_load_2d(l0 + off, txlo, bar, kb * kTileK, r0);
  }
}

// MMAs of one stage into accumulator column `d`: every M-tile holding rows
// (and, SPLIT, its remainder terms into the same accumulator).
template <bool SPLIT>
__device__ __forceinline__ void tc_mma_stage(const uint8_t* st, uint32_t d, const TcParams& p, int m,
                                             uint32_t idesc, bool first) {
  const uint64_t dw = ptx::smem_desc_sw128(st + p.w_off);
  for (int t = 0; t < p.mt && t * 128 < m; ++t) {
    const uint8_t* xt = st + t * p.xr;
    const uint64_t dx = ptx::smem_desc_sw128(xt);
    const uint64_t dl = ptx::smem_desc_sw128(xt + p.mt * p.xr);
    const uint32_t dt = d + (uint32_t)(t * p.bw);
#pragma unroll
    for (int k = 0; k < kTileK / 16; ++k) {
      ptx::mma_bf16(dt, dx + 2ull * k, dw + 2ull * k, idesc, (!first || k > 0) ? 1u : 0u);
      if (SPLIT) ptx::mma_bf16(dt, dl + 2ull * k, dw + 2ull * k, idesc, 1u);
    }
  }
}

// ---------------------------------------------------------------------------
// Panel mode.  Panel layout: K block r of the unit at r * 1024 bytes, rows 0..7
// of the 128-byte-swizzled K-major tile (rows past m unused); the remainder
// terms at panel_kb * 1024.  An M = 128 operand read from block r spans the
// following 15 KiB (later blocks, the next panel, or the tail slack): those
// rows only feed accumulator rows that are discarded.
// ---------------------------------------------------------------------------
// 1 / rms of each row (m <= 8), by the 128 epilogue threads (et = 0..127).
__device__ __forceinline__ void tc_panel_inv(const TcParams& p, int m, int et, float* red, float* inv) {
  const int lane = et & 31, w = et >> 5;
  for (int j = 0; j < m; ++j) {
    const float* h = p.nsrc + (size_t)(p.rows ? p.rows[j] : j) * p.K;
    float ss = 0.f;
    for (int e0 = 0; e0 < p.K; e0 += 16 * 512) {
      float4 x[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const int e = e0 + (et + k * 128) * 4;
        x[k] = e < p.K ? *reinterpret_cast<const float4*>(h + e) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < 16; ++k) ss += x[k].x * x[k].x + x[k].y * x[k].y + x[k].z * x[k].z + x[k].w * x[k].w;
    }
    ss = warp_sum(ss);
    if (lane == 0) red[j * 4 + w] = ss;
  }
  epi_bar();
  if (et < m) inv[et] = rsqrtf(((red[et * 4] + red[et * 4 + 1]) + (red[et * 4 + 2] + red[et * 4 + 3])) / (float)p.K + p.neps);
  epi_bar();
}

// The panel of K blocks [kb0, kb1) for rows j < m, then a proxy fence so that
// the tensor core sees it.  Each thread takes float4 groups (row, column) with
// all loads issued before the stores.
template <bool SPLIT>
__device__ __forceinline__ void tc_panel_write(const TcParams& p, uint8_t* panel, int m, int kb0, int kb1, int et,
                                               const float* inv) {
  const int n4 = (kb1 - kb0) * 16;   // float4 groups per row
  const int total = m * n4;
  for (int i0 = et; i0 < total; i0 += 4 * 128) {
    float4 x[4], g[4];
    int jj[4], qq[4];
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int i = i0 + b * 128;
      jj[b] = i < total ? i / n4 : -1;
      qq[b] = i - (jj[b] < 0 ? 0 : jj[b]) * n4;
      if (jj[b] >= 0) {
        const int c = kb0 * kTileK + qq[b] * 4;
        x[b] = *reinterpret_cast<const float4*>(p.nsrc + (size_t)(p.rows ? p.rows[jj[b]] : jj[b]) * p.K + c);
        g[b] = *reinterpret_cast<const float4*>(p.ngamma + c);
      }
    }
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      if (jj[b] < 0) continue;
      const int j = jj[b], r = qq[b] >> 4, q = qq[b] & 15;
      const float iv = inv[j];
      const float y[4] = {x[b].x * iv * g[b].x, x[b].y * iv * g[b].y, x[b].z * iv * g[b].z, x[b].w * iv * g[b].w};
      uint32_t hi[2], lo[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const bf16 a = from_f<bf16>(y[2 * u]), c2 = from_f<bf16>(y[2 * u + 1]);
        hi[u] = (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(c2) << 16);
        if (SPLIT) {
          const bf16 la = from_f<bf16>(y[2 * u] - to_f(a)), lc = from_f<bf16>(y[2 * u + 1] - to_f(c2));
          lo[u] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lc) << 16);
        }
      }
      // row j of K block r: 16-byte chunk q / 2 of the row at chunk (q / 2) ^ j
      const uint32_t off = (uint32_t)r * 1024u + (uint32_t)j * 128u + (uint32_t)((((q >> 1) ^ j) & 7) << 4) +
                           (uint32_t)((q & 1) * 8);
      *reinterpret_cast<uint2*>(panel + off) = make_uint2(hi[0], hi[1]);
      if (SPLIT) *reinterpret_cast<uint2*>(panel + (size_t)p.panel_kb * 1024 + off) = make_uint2(lo[0], lo[1]);
    }
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Largest K the single-pass first panel handles (one float4 per thread per
// 512 columns, 16 per thread).
constexpr int kPanelFirstMaxK = 16 * 512;

// The first unit's panel in one pass over each row: every thread loads its
// 16 float4 of row j (the loads of the sum of squares), the sum is reduced
// across the 4 epilogue warps, and the thread then writes the panel entries
// of the unit's K range [kb0, kb1) that it already holds, scaled by 1 / rms
// and by the gains staged in shared memory (gst, from column kb0 * 64).  The
// arithmetic (order of the squares, of the reduction and of the products) is
// that of tc_panel_inv followed by tc_panel_write.  row_of[j] holds the
// source row of panel row j.
template <bool SPLIT>
__device__ __forceinline__ void tc_panel_first(const TcParams& p, uint8_t* panel, int m, int kb0, int kb1, int et,
                                               const int* row_of, const float* gst, float* red, float* inv) {
  const int lane = et & 31, w = et >> 5;
  const int c_lo = kb0 * kTileK, c_hi = kb1 * kTileK;
  for (int j = 0; j < m; ++j) {
    const float* h = p.nsrc + (size_t)row_of[j] * p.K;
    float4 x[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int e = (et + k * 128) * 4;
      x[k] = e < p.K ? *reinterpret_cast<const float4*>(h + e) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float ss = 0.f;
#pragma unroll
    for (int k = 0; k < 16; ++k) ss += x[k].x * x[k].x + x[k].y * x[k].y + x[k].z * x[k].z + x[k].w * x[k].w;
    ss = warp_sum(ss);
    if (lane == 0) red[j * 4 + w] = ss;
    epi_bar();
    const float iv = rsqrtf(((red[j * 4] + red[j * 4 + 1]) + (red[j * 4 + 2] + red[j * 4 + 3])) / (float)p.K + p.neps);
    if (et == 0) inv[j] = iv;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int e = (et + k * 128) * 4;
      if (e < c_lo || e >= c_hi) continue;
      const int c = e - c_lo, r = c >> 6, q = (c & 63) >> 2;
      const float4 g = *reinterpret_cast<const float4*>(gst + c);
      const float y[4] = {x[k].x * iv * g.x, x[k].y * iv * g.y, x[k].z * iv * g.z, x[k].w * iv * g.w};
      uint32_t hi[2], lo[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const bf16 a = from_f<bf16>(y[2 * u]), c2 = from_f<bf16>(y[2 * u + 1]);
        hi[u] = (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(c2) << 16);
        if (SPLIT) {
          const bf16 la = from_f<bf16>(y[2 * u] - to_f(a)), lc = from_f<bf16>(y[2 * u + 1] - to_f(c2));
          lo[u] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lc) << 16);
        }
      }
      const uint32_t off = (uint32_t)r * 1024u + (uint32_t)j * 128u + (uint32_t)((((q >> 1) ^ j) & 7) << 4) +
                           (uint32_t)((q & 1) * 8);
      *reinterpret_cast<uint2*>(panel + off) = make_uint2(hi[0], hi[1]);
      if (SPLIT) *reinterpret_cast<uint2*>(panel + (size_t)p.panel_kb * 1024 + off) = make_uint2(lo[0], lo[1]);
    }
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// MMAs of one stage in panel mode: weights from the stage, activations (one
// M-tile, and SPLIT the remainder terms) from panel block `pb`.
template <bool SPLIT>
__device__ __forceinline__ void tc_mma_panel(const uint8_t* st, const uint8_t* pb, uint32_t d, const TcParams& p,
                                             uint32_t idesc, bool first) {
  const uint64_t dw = ptx::smem_desc_sw128(st);
  const uint64_t dx = ptx::smem_desc_sw128(pb);
  const uint64_t dl = ptx::smem_desc_sw128(pb + (size_t)p.panel_kb * 1024);
#pragma unroll
  for (int k = 0; k < kTileK / 16; ++k) {
    ptx::mma_bf16(d, dx + 2ull * k, dw + 2ull * k, idesc, (!first || k > 0) ? 1u : 0u);
    if (SPLIT) ptx::mma_bf16(d, dl + 2ull * k, dw + 2ull * k, idesc, 1u);
  }
}

// ---------------------------------------------------------------------------
// Epilogue of row j, accumulator columns c..c+3 of a tile (`v`), with the
// partner columns `vp` where the epilogue pairs columns (SwiGLU: the up rows
// bw/2 further on; QKV: the other half of each rotate-half pair, hd/2 further).
// ---------------------------------------------------------------------------
template <int EPI>
__device__ __forceinline__ int tc_partner_off(const TcParams& p) {
  return EPI == EPI_SWIGLU ? (p.bw >> 1) : (EPI == EPI_QKV ? (p.hd >> 1) : 0);
}
// Work items of one tile's epilogue: (row, group of 4 primary columns).
template <int EPI>
__device__ __forceinline__ int tc_groups(const TcParams& p) {
  return EPI == EPI_SWIGLU || EPI == EPI_QKV ? p.bw / 8 : p.bw / 4;
}
template <int EPI>
__device__ __forceinline__ int tc_group_col(const TcParams& p, int g) {
  if (EPI == EPI_QKV) {
    const int per = p.hd >> 3;   // groups in the low half of a head
    return (g / per) * p.hd + (g % per) * 4;
  }
  return g * 4;
}

__device__ __forceinline__ uint2 pack4_bf16(const float* y) {
  return make_uint2((uint32_t)__bfloat16_as_ushort(from_f<bf16>(y[0])) |
                        ((uint32_t)__bfloat16_as_ushort(from_f<bf16>(y[1])) << 16),
                    (uint32_t)__bfloat16_as_ushort(from_f<bf16>(y[2])) |
                        ((uint32_t)__bfloat16_as_ushort(from_f<bf16>(y[3])) << 16));
}

template <int EPI, bool SPLIT>
__device__ __forceinline__ void tc_apply4(const TcParams& p, int tile, int j, int c, const float* v, const float* vp,
                                          const float* rs) {
  if (EPI == EPI_SWIGLU) {
    const int f0 = tile * (p.bw >> 1) + c;
    if (f0 + 4 <= p.N) {   // one 8-byte store (N % 8 == 0, c % 4 == 0)
      uint32_t hi[2], lo[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const float a0 = silu_f(v[2 * u]) * vp[2 * u], a1 = silu_f(v[2 * u + 1]) * vp[2 * u + 1];
        const bf16 b0 = from_f<bf16>(a0), b1 = from_f<bf16>(a1);
        hi[u] = (uint32_t)__bfloat16_as_ushort(b0) | ((uint32_t)__bfloat16_as_ushort(b1) << 16);
        if (SPLIT) {
          const bf16 l0 = from_f<bf16>(a0 - to_f(b0)), l1 = from_f<bf16>(a1 - to_f(b1));
          lo[u] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
        }
      }
      *reinterpret_cast<uint2*>(p.out_act + (size_t)j * p.N + f0) = make_uint2(hi[0], hi[1]);
      if (SPLIT) *reinterpret_cast<uint2*>(p.out_act_lo + (size_t)j * p.N + f0) = make_uint2(lo[0], lo[1]);
      return;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int f = f0 + i;
      if (f < p.N) {
        const float a = silu_f(v[i]) * vp[i];
        const bf16 hi = from_f<bf16>(a);
        p.out_act[(size_t)j * p.N + f] = hi;
        if (SPLIT) p.out_act_lo[(size_t)j * p.N + f] = from_f<bf16>(a - to_f(hi));
      }
    }
  } else if (EPI == EPI_QKV) {
    const int hd = p.hd, half = hd >> 1;
    const int n0 = tile * p.bw + c;
    if (n0 >= p.N) return;   // heads are whole: a group and its partner are in or out together
    const int head = n0 / hd, e0 = n0 - head * hd;
    const int seq = p.rows ? p.rows[j] : j;
    const int pos = p.len[seq];
    const int cpos = p.cache_len[seq];
    float x[4], xp[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[i] = v[i] + (p.bias ? p.bias[n0 + i] : 0.f);
      xp[i] = vp[i] + (p.bias ? p.bias[n0 + half + i] : 0.f);
    }
    if (head < p.nq + p.nkv) {
      const float* co = p.rope_cos + (size_t)pos * half + e0;
      const float* si = p.rope_sin + (size_t)pos * half + e0;
      float lo[4], hi[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        lo[i] = x[i] * co[i] - xp[i] * si[i];
        hi[i] = xp[i] * co[i] + x[i] * si[i];
      }
      if (head < p.nq) {
        float* q = p.q_out + (size_t)j * p.nq * hd + n0;
        *reinterpret_cast<float4*>(q) = make_float4(lo[0], lo[1], lo[2], lo[3]);
        *reinterpret_cast<float4*>(q + half) = make_float4(hi[0], hi[1], hi[2], hi[3]);
      } else {
        bf16* k = p.kc + kv_offset(p.seq_off, p.cap, seq, p.nkv, hd, head - p.nq, cpos) + e0;
        *reinterpret_cast<uint2*>(k) = pack4_bf16(lo);
        *reinterpret_cast<uint2*>(k + half) = pack4_bf16(hi);
      }
    } else {
      const int g = head - p.nq - p.nkv;
      bf16* vv = p.vc + kv_offset(p.seq_off, p.cap, seq, p.nkv, hd, g, cpos) + e0;
      float* pl = p.pool ? p.pool + (size_t)seq * p.nkv * hd + g * hd + e0 : nullptr;
      *reinterpret_cast<uint2*>(vv) = pack4_bf16(x);
      *reinterpret_cast<uint2*>(vv + half) = pack4_bf16(xp);
      if (pl) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          pl[i] += to_f(from_f<bf16>(x[i]));
          pl[half + i] += to_f(from_f<bf16>(xp[i]));
        }
      }
    }
  } else {
    const int n0 = tile * p.bw + c;
    float* dst;
    float w[4];
    if (EPI == EPI_STORE_F32) {
      dst = p.out_f32 + (size_t)j * p.N + n0;
#pragma unroll
      for (int i = 0; i < 4; ++i) w[i] = v[i];
    } else {
      const int seq = p.rows ? p.rows[j] : j;
      dst = p.resid_dst + (size_t)seq * p.N + n0;
#pragma unroll
      for (int i = 0; i < 4; ++i) w[i] = rs[i] + v[i];
    }
    if (n0 + 4 <= p.N) {   // one 16-byte store (N % 4 == 0, c % 4 == 0)
      *reinterpret_cast<float4*>(dst) = make_float4(w[0], w[1], w[2], w[3]);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (n0 + i < p.N) dst[i] = w[i];
    }
  }
}

// Position (in float4 units) of row j's 4-column group at column c in a
// workspace slot.  Up to 16 rows a slot is row-major (the groups of a row
// contiguous: the few rows' items are read group by group); above, group-major
// (a group's rows contiguous: the 32 lanes of a warp hold 32 rows of an
// accumulator column block, and store 512 contiguous bytes per group).
__device__ __forceinline__ size_t tc_ws_idx(const TcParams& p, int j, int c) {
  return p.rows_max <= 16 ? (size_t)j * (p.bw >> 2) + (c >> 2) : (size_t)(c >> 2) * p.rows_max + j;
}

// One epilogue item (row j, 4-column group at c of `tile`): the partials of
// all K splits (and of the partner columns) are summed in split order, eight
// splits' loads in flight at a time, and the epilogue is applied.
template <int EPI, bool SPLIT>
__device__ __forceinline__ void tc_fix_item(const TcParams& p, int tile, int j, int c) {
  const int po = tc_partner_off<EPI>(p);
  const size_t sstride = (size_t)p.n_tiles * p.rows_max * p.bw / 4;   // one split's slots (float4)
  const size_t pstride = tc_ws_idx(p, j, c + po) - tc_ws_idx(p, j, c);
  const float4* sl = reinterpret_cast<const float4*>(p.ws + (size_t)tile * p.rows_max * p.bw) + tc_ws_idx(p, j, c);
  float v[4] = {0.f, 0.f, 0.f, 0.f}, vp[4] = {0.f, 0.f, 0.f, 0.f}, rs[4] = {0.f, 0.f, 0.f, 0.f};
  if (EPI == EPI_RESID) {
    const int seq = p.rows ? p.rows[j] : j;
    const int n0 = tile * p.bw + c;
    const float* src = p.resid_src + (size_t)seq * p.N + n0;
    if (n0 + 4 <= p.N) {
      const float4 r4 = *reinterpret_cast<const float4*>(src);
      rs[0] = r4.x; rs[1] = r4.y; rs[2] = r4.z; rs[3] = r4.w;
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (n0 + i < p.N) rs[i] = src[i];
    }
  }
  for (int s0 = 0; s0 < p.splits; s0 += 8) {
    float4 x[8], y[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (s0 + k < p.splits) {
        x[k] = __ldcg(sl + (size_t)(s0 + k) * sstride);
        if (po) y[k] = __ldcg(sl + (size_t)(s0 + k) * sstride + pstride);
      }
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (s0 + k < p.splits) {
        v[0] += x[k].x; v[1] += x[k].y; v[2] += x[k].z; v[3] += x[k].w;
        if (po) {
          vp[0] += y[k].x; vp[1] += y[k].y; vp[2] += y[k].z; vp[3] += y[k].w;
        }
      }
    }
  }
  tc_apply4<EPI, SPLIT>(p, tile, j, c, v, vp, rs);
}

// ---------------------------------------------------------------------------
// Epilogue of one unit by the four epilogue warps (128 threads).  Warp w reads
// TMEM lanes 32*(w%4).. (rows of each M-tile) and writes the unit's
// accumulator rows j < m to its workspace slot; the accumulator is released
// (tempty) right after.  The CTA that completes a tile (the last of its K
// splits, or the only one) then applies the epilogue with all 128 threads over
// (row, 4-column group) items, summing the splits' slots in split order
// (deterministic).  With p.defer every unit stops after staging its slot,
// except a SwiGLU GEMM with a single K split, which applies its epilogue
// directly.
// ---------------------------------------------------------------------------
template <int EPI, bool SPLIT>
__device__ __forceinline__ void tc_epilogue_unit(const TcParams& p, int u, int m, uint32_t tacc, uint64_t* tempty,
                                                 int* last_flag) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3;   // TMEM lane quarter this warp may access
  const int tile = u % p.n_tiles;
  if (EPI == EPI_SWIGLU && p.defer && p.splits == 1) {
    // One K split (larger batches): SwiGLU straight from the accumulator, gate
    // column c and up column c + bw/2 of the same row, with no workspace and no
    // fixup kernel (the same arithmetic as tc_apply4 on a single partial).
    const int h = p.bw >> 1;
    for (int t = 0; t < p.mt; ++t) {
      if (t * 128 + q * 32 >= m) continue;   // warp-uniform
      const int j = t * 128 + q * 32 + lane;
      const uint32_t ta = tacc + ((uint32_t)(q * 32) << 16) + (uint32_t)(t * p.bw);
      for (int c0 = 0; c0 < h; c0 += 16) {
        float g[16], up[16];
        ptx::tmem_ld16(ta + c0, g);
        ptx::tmem_ld16(ta + h + c0, up);
        if (j >= m) continue;
        const int f0 = tile * h + c0;
        uint32_t hi[8], lo[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float a0 = silu_f(g[2 * i]) * up[2 * i], a1 = silu_f(g[2 * i + 1]) * up[2 * i + 1];
          const bf16 b0 = from_f<bf16>(a0), b1 = from_f<bf16>(a1);
          hi[i] = (uint32_t)__bfloat16_as_ushort(b0) | ((uint32_t)__bfloat16_as_ushort(b1) << 16);
          if (SPLIT) {
            const bf16 l0 = from_f<bf16>(a0 - to_f(b0)), l1 = from_f<bf16>(a1 - to_f(b1));
            lo[i] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
          }
        }
        bf16* dst = p.out_act + (size_t)j * p.N + f0;
        bf16* dlo = SPLIT ? p.out_act_lo + (size_t)j * p.N + f0 : nullptr;
        if (f0 + 16 <= p.N) {   // 32 bytes, 16-byte aligned (N % 8 == 0)
          reinterpret_cast<uint4*>(dst)[0] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          reinterpret_cast<uint4*>(dst)[1] = make_uint4(hi[4], hi[5], hi[6], hi[7]);
          if (SPLIT) {
            reinterpret_cast<uint4*>(dlo)[0] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            reinterpret_cast<uint4*>(dlo)[1] = make_uint4(lo[4], lo[5], lo[6], lo[7]);
          }
        } else {
          for (int i = 0; i < 16 && f0 + i < p.N; ++i) {
            const uint32_t w = hi[i >> 1] >> ((i & 1) * 16);
            dst[i] = __ushort_as_bfloat16((unsigned short)(w & 0xFFFFu));
            if (SPLIT) dlo[i] = __ushort_as_bfloat16((unsigned short)((lo[i >> 1] >> ((i & 1) * 16)) & 0xFFFFu));
          }
        }
      }
    }
    ptx::tc_fence_before();
    if (lane == 0) ptx::mbar_arrive(tempty);
    return;
  }
  float4* slot = reinterpret_cast<float4*>(p.ws + (size_t)u * p.rows_max * p.bw);
  for (int t = 0; t < p.mt; ++t) {
    if (t * 128 + q * 32 >= m) continue;   // warp-uniform
    const int j = t * 128 + q * 32 + lane;
    const uint32_t ta = tacc + ((uint32_t)(q * 32) << 16) + (uint32_t)(t * p.bw);
    for (int c0 = 0; c0 < p.bw; c0 += 64) {
      float v[64];
      ptx::tmem_ld64(ta + c0, v);
      if (j < m) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          __stcg(slot + tc_ws_idx(p, j, c0 + 4 * i), make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]));
      }
    }
  }
  ptx::tc_fence_before();
  if (lane == 0) ptx::mbar_arrive(tempty);
  if (p.defer) return;   // gemm_fix_kernel sums the splits
  epi_bar();
  const int et = threadIdx.x & 127;
  if (et == 0) {
    // release of this CTA's slot (stored before the barrier) and, for the
    // last arriver, acquire of the other splits' slots
    int last = 1;
    if (p.splits > 1) {
      const int old = ptx::atom_add_acq_rel(&p.ctr[tile], 1);
      last = old == p.splits - 1;
      if (last) p.ctr[tile] = 0;   // re-armed for a later launch
    }
    *last_flag = last;
  }
  epi_bar();
  if (*last_flag) {
    const int ng = tc_groups<EPI>(p);
    const int items = m * ng;
    for (int it = et; it < items; it += 128) {   // one item per thread per round
      const int j = it / ng;
      tc_fix_item<EPI, SPLIT>(p, tile, j, tc_group_col<EPI>(p, it - j * ng));
    }
  }
  epi_bar();
}

// GEMM shapes: which = 0 qkv, 1 o, 2 gate_up, 3 down; tiles of bw features
// (gate/up: bw/2 features, each with its gate and up rows)
inline void gemm_shape(const Ctx& c, int which, int* N, int* K, int* tiles) {
  const int bw = c.tc_bw;
  switch (which) {
    case 0: *N = c.qkvN; *K = c.d; *tiles = (c.qkvN + bw - 1) / bw; break;
    case 1: *N = c.d; *K = c.qd; *tiles = (c.d + bw - 1) / bw; break;
    case 2: *N = c.F; *K = c.d; *tiles = (c.F + bw / 2 - 1) / (bw / 2); break;
    default: *N = c.d; *K = c.F; *tiles = (c.d + bw - 1) / bw; break;
  }
}

}  // namespace buddy

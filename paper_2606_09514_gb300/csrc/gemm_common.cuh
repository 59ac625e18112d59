// Shared pieces of the tensor-core GEMM (gemm_tc.cu) and the per-layer
// persistent kernel (layer_kernel.cu): tile constants, parameters of one GEMM,
// and the epilogues applied to a 128-feature x 16-row block of results.
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace buddy {

constexpr int kTcThreads = 192;
constexpr int kTcMaxStages = 16;
constexpr int kTileK = 64;
constexpr uint32_t kTileABytes = 128 * kTileK * 2;   // 16 KiB weight tile
constexpr uint64_t kWaitLimitNs = 4000000000ull;     // 4 s

struct TcParams {
  int N, K;
  int n_tiles, splits, kb_total, kb_per_split, units;
  int bn_max, stages;
  uint32_t stage_bytes, tmem_cols;
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
  const int32_t* len;
  const int64_t* seq_off;
  const int32_t* cap;
  bf16* kc;
  bf16* vc;
  float* q_out;
  float* pool;
  int nq, nkv, hd;
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

template <int EPI, bool SPLIT>
__device__ __forceinline__ void apply_epilogue(const TcParams& p, int tile, int row, int c0, int m,
                                               const float* v, float* xch) {
  if (EPI == EPI_QKV) {
    // a 128-row tile holds whole heads (hd = 64 or 128): RoPE partners are
    // rows of the same tile, exchanged through shared memory
#pragma unroll
    for (int i = 0; i < 16; ++i) xch[row * 17 + i] = v[i];
    epi_bar();
    const int nf = tile * 128 + row;
    if (nf < p.N) {
      const int hd = p.hd, half = hd >> 1;
      const int head = nf / hd, e = nf - head * hd;
      const bool lowh = e < half;
      const int pr = lowh ? row + half : row - half;
      const int ep = lowh ? e : e - half;
      const float b0 = p.bias ? p.bias[nf] : 0.f;
      const float bp = p.bias ? p.bias[lowh ? nf + half : nf - half] : 0.f;
      const int kvd = p.nkv * hd;
      for (int i = 0; i < 16; ++i) {
        const int j = c0 + i;
        if (j >= m) break;
        const int seq = p.rows ? p.rows[j] : j;
        const int pos = p.len[seq];
        const float x = v[i] + b0;
        if (head < p.nq + p.nkv) {
          const float xp = xch[pr * 17 + i] + bp;
          const float co = p.rope_cos[(size_t)pos * half + ep], si = p.rope_sin[(size_t)pos * half + ep];
          const float y = lowh ? x * co - xp * si : x * co + xp * si;
          if (head < p.nq) {
            p.q_out[(size_t)j * p.nq * hd + nf] = y;
          } else {
            const int g = head - p.nq;
            p.kc[kv_offset(p.seq_off, p.cap, seq, p.nkv, hd, g, pos) + e] = from_f<bf16>(y);
          }
        } else {
          const int g = head - p.nq - p.nkv;
          const bf16 vs = from_f<bf16>(x);
          p.vc[kv_offset(p.seq_off, p.cap, seq, p.nkv, hd, g, pos) + e] = vs;
          if (p.pool) p.pool[(size_t)seq * kvd + g * hd + e] += to_f(vs);
        }
      }
    }
    epi_bar();
  } else if (EPI == EPI_SWIGLU) {
    // rows 0..63: gate of feature f = tile*64 + row; rows 64..127: up of the same f
    const bool up = row >= 64;
    const int r = row & 63;
    if (up) {
#pragma unroll
      for (int i = 0; i < 16; ++i) xch[r * 17 + i] = v[i];
    }
    epi_bar();
    if (!up) {
      const int f = tile * 64 + r;
      if (f < p.N) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int j = c0 + i;
          if (j < m) {
            const float a = silu_f(v[i]) * xch[r * 17 + i];
            const bf16 hi = from_f<bf16>(a);
            p.out_act[(size_t)j * p.N + f] = hi;
            if (SPLIT) p.out_act_lo[(size_t)j * p.N + f] = from_f<bf16>(a - to_f(hi));
          }
        }
      }
    }
    epi_bar();
  } else {
    const int nf = tile * 128 + row;
    if (nf >= p.N) return;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int j = c0 + i;
      if (j >= m) break;
      if (EPI == EPI_STORE_F32) {
        p.out_f32[(size_t)j * p.N + nf] = v[i];
      } else {
        const int seq = p.rows ? p.rows[j] : j;
        const size_t o = (size_t)seq * p.N + nf;
        p.resid_dst[o] = p.resid_src[o] + v[i];
      }
    }
  }
}

// GEMM shapes: which = 0 qkv, 1 o, 2 gate_up, 3 down
inline void gemm_shape(const Ctx& c, int which, int* N, int* K, int* tiles) {
  switch (which) {
    case 0: *N = c.qkvN; *K = c.d; *tiles = (c.qkvN + 127) / 128; break;
    case 1: *N = c.d; *K = c.qd; *tiles = (c.d + 127) / 128; break;
    case 2: *N = c.F; *K = c.d; *tiles = (c.F + 63) / 64; break;
    default: *N = c.d; *K = c.F; *tiles = (c.d + 127) / 128; break;
  }
}

}  // namespace buddy

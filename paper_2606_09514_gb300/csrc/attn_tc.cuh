// Decode attention on the tensor cores (bf16 caches, head dim 64 or 128, at
// most 8 query heads per KV head).  Same work decomposition and results as the
// SIMT work loop in attn_common.cuh (items = row x KV head x span of P
// positions, split spans merged in span order by the last CTA to finish), but
// inside a span each of the four warps streams its own 32-position chunks:
//
//   * K and V rows of the chunk are copied with 16-byte cp.async into the
//     warp's double buffer (rows padded by 16 bytes: ldmatrix conflict-free);
//   * logits S = Q K^T with mma.sync m16n8k16 (bf16 in, fp32 accumulate): the
//     query heads are the 16 rows of A (heads >= G are zero), K rows feed B
//     through ldmatrix;
//   * online softmax on the accumulator fragments (quad shuffles per row);
//   * O += P V with the probabilities taken straight from the S fragments as
//     the A operand and V through ldmatrix.trans.
//
// With SPLIT (the first block, which feeds the router) the scaled queries and
// the probabilities are each given as bf16 hi + lo and every product is issued
// for both terms, so the contractions carry ~16 mantissa bits; otherwise one
// bf16 term each.  The four warps' running (max, sum, output) are combined in
// shared memory.
#pragma once

#include <cuda_runtime.h>

#include "attn_common.cuh"
#include "common.cuh"

namespace buddy {

constexpr int kTcaChunk = 32;     // positions per warp chunk
constexpr int kTcaWarps = 4;
constexpr int kTcaThreads = 32 * kTcaWarps;

template <int HD>
__host__ __device__ constexpr size_t attn_tc_smem_fixed() {
  // per warp: two buffers of K and V rows, each row padded by 8 bf16
  return (size_t)kTcaWarps * 2 * 2 * kTcaChunk * (HD + 8) * 2;
}
inline size_t attn_tc_smem_bytes(int hd, int max_rows) {
  const size_t fixed = hd == 128 ? attn_tc_smem_fixed<128>() : attn_tc_smem_fixed<64>();
  return fixed + (size_t)(max_rows + 1) * 4 + 8 + (size_t)max_rows * 16;
}

namespace tca {

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
         ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
}
// hi = bf16 pair of (a, b); lo = bf16 pair of the remainders
__device__ __forceinline__ void split_pack(float a, float b, uint32_t& hi, uint32_t& lo) {
  const bf16 ha = __float2bfloat16_rn(a), hb = __float2bfloat16_rn(b);
  hi = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
  lo = pack_bf16(a - __bfloat162float(ha), b - __bfloat162float(hb));
}
__device__ __forceinline__ void ldsm_x4(const void* p, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}
__device__ __forceinline__ void ldsm_x4_t(const void* p, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}
// D (16x8 fp32) += A (16x16 bf16, rows 8..15 zero) * B (16x8 bf16).  Only
// rows 0..7 are kept (d0, d1 of this thread); rows 8..15 go to scratch z.
__device__ __forceinline__ void mma16816(float& d0, float& d1, float (&z)[2], uint32_t a0, uint32_t a2, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d0), "+f"(d1), "+f"(z[0]), "+f"(z[1])
      : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
}

}  // namespace tca

// Processes this CTA's share of one layer's attention (kTcaThreads threads).
// Smem layout: per-warp K/V double buffers, then the row prefix and the rows'
// cache offsets, positions and head strides.  `sc` is 32 floats of scratch.
template <int HD, bool SPLIT>
__device__ __forceinline__ void attn_tc_run(const AttnArgs<bf16>& A, int cta, int ncta, uint8_t* smem, float* sc,
                                            bool pdl) {
  static_assert(HD == 64 || HD == 128, "HD");
  constexpr int KROW = HD + 8;                    // padded row (elements)
  constexpr int KSTEPS = HD / 16;                 // k-steps of the logits
  constexpr int DT = HD / 8;                      // output n-tiles
  constexpr int V16 = HD / 8;                     // 16-byte pieces per row
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t* rows = A.rows;
  const int nq = A.nq, nkv = A.nkv, G = nq / nkv;
  const int aborted = *reinterpret_cast<const volatile int32_t*>(A.status + 1);
  const int m = A.count ? *A.count : A.n;
  if (aborted != 0 || m <= 0) {
    if (pdl) pdl_wait();
    return;
  }
  bf16* wbuf = reinterpret_cast<bf16*>(smem) + (size_t)warp * 2 * 2 * kTcaChunk * KROW;   // this warp's buffers
  int* pref = reinterpret_cast<int*>(smem + attn_tc_smem_fixed<HD>());
  int64_t* rbase = reinterpret_cast<int64_t*>((reinterpret_cast<uintptr_t>(pref + m + 1) + 7) & ~uintptr_t(7));
  int* rnp = reinterpret_cast<int*>(rbase + m);
  int* rhs = rnp + m;
  float* mw = reinterpret_cast<float*>(smem);                   // merge: [warps][8] max
  float* lw = mw + kTcaWarps * 8;                               //        [warps][8] sum
  float* ow = lw + kTcaWarps * 8;                               //        [warps][8][HD] output
  int* last_s_p = reinterpret_cast<int*>(sc + 24);
  int* span_s_p = reinterpret_cast<int*>(sc + 25);

  // positions per row and their total -> span length P (as attn_run)
  if (warp == 0) {
    long long tot = 0;
    for (int j = lane; j < m; j += 32) {
      const int i = rows ? rows[j] : j;
      const int np = A.len[i] + 1;
      rnp[j] = np;
      rbase[j] = A.seq_off[i] * nkv * HD;
      rhs[j] = A.cap[i] * HD;
      pref[j + 1] = np;
      tot += np;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    __syncwarp();
    // about one item per CTA; a span is a multiple of the four warps' chunks
    const long long want = (tot * nkv + ncta - 1) / ncta;
    constexpr int kQ = kTcaChunk * kTcaWarps;
    const int P0 = (int)min((long long)kMaxSpan, max((long long)kQ, want));
    const int P = (P0 + kQ - 1) / kQ * kQ;
    int carry = 0;
    for (int b = 0; b < m; b += 32) {
      const int j = b + lane;
      int ns = 0;
      if (j < m) ns = (pref[j + 1] + P - 1) / P;
      int x = ns;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      __syncwarp();
      if (j < m) pref[j + 1] = carry + x;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) {
      pref[0] = 0;
      *span_s_p = P;
    }
  }
  __syncthreads();
  const int P = *span_s_p;
  const int total = pref[m] * nkv;
  const float scale = rsqrtf((float)HD);
  bool waited = !pdl;
  const int h0 = lane >> 2, c2 = (lane & 3) * 2;   // fragment row (head) and column pair

  for (int item = cta; item < total; item += ncta) {
    const int g = item % nkv;
    const int js = item / nkv;
    int lo = 0, hi = m;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pref[mid] <= js) lo = mid;
      else hi = mid;
    }
    const int j = lo, sp = js - pref[j];
    const int npos = rnp[j];
    const int nsp = pref[j + 1] - pref[j];
    const int s0 = sp * P, s1 = min(npos, s0 + P);
    const int nch = (s1 - s0 + kTcaChunk - 1) / kTcaChunk;   // chunks of the span
    const int64_t kvo = rbase[j] + (int64_t)g * rhs[j];
    const bf16* Kbase = A.Kc + kvo;
    const bf16* Vbase = A.Vc + kvo;

    // this warp's chunks: c = warp, warp + 4, ...
    auto issue = [&](int c, int buf) {
      const int p0 = s0 + c * kTcaChunk, cnt = min(kTcaChunk, s1 - p0);
      bf16* Kd = wbuf + (size_t)buf * 2 * kTcaChunk * KROW;
      bf16* Vd = Kd + kTcaChunk * KROW;
      for (int x = lane; x < cnt * V16; x += 32) {
        const int p = x / V16, s = x - p * V16;
        cp_async16(Kd + p * KROW + s * 8, Kbase + (size_t)(p0 + p) * HD + s * 8);
        cp_async16(Vd + p * KROW + s * 8, Vbase + (size_t)(p0 + p) * HD + s * 8);
      }
      // rows past the span end: zero V (their probabilities are 0, and 0 times
      // stale shared memory could be NaN); K is masked on the logits
      for (int x = cnt * V16 + lane; x < kTcaChunk * V16; x += 32) {
        const int p = x / V16, s = x - p * V16;
        *reinterpret_cast<uint4*>(Vd + p * KROW + s * 8) = make_uint4(0u, 0u, 0u, 0u);
      }
      cp_async_commit();
    };
    const int c_first = warp;
    const bool has_work = c_first < nch;
    if (!waited) {
      // a chunk without the new token (position npos - 1) may be copied first
      const bool has_new = has_work && s0 + (c_first + 1) * kTcaChunk >= npos;
      if (has_work && !has_new) issue(c_first, 0);
      pdl_wait();
      pdl_trigger();
      waited = true;
      if (has_work && has_new) issue(c_first, 0);
    } else if (has_work) {
      issue(c_first, 0);
    }
    // query fragments: rows = heads (h0 < G), columns = dims; scaled
    uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
    {
      const float* qj = A.q + (size_t)j * nq * HD + (size_t)g * G * HD + (size_t)h0 * HD;
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        float x0 = 0.f, x1 = 0.f, x2 = 0.f, x3 = 0.f;
        if (h0 < G) {
          const float2 a = *reinterpret_cast<const float2*>(qj + kk * 16 + c2);
          const float2 b = *reinterpret_cast<const float2*>(qj + kk * 16 + 8 + c2);
          x0 = a.x * scale; x1 = a.y * scale; x2 = b.x * scale; x3 = b.y * scale;
        }
        if (SPLIT) {
          tca::split_pack(x0, x1, qh[kk][0], ql[kk][0]);
          tca::split_pack(x2, x3, qh[kk][1], ql[kk][1]);
        } else {
          qh[kk][0] = tca::pack_bf16(x0, x1);
          qh[kk][1] = tca::pack_bf16(x2, x3);
        }
      }
    }
    float mrun = -INFINITY, lrun = 0.f;
    float o[DT][2];
    float z[2] = {0.f, 0.f};   // rows 8..15 of every product (padding heads)
#pragma unroll
    for (int t = 0; t < DT; ++t) o[t][0] = o[t][1] = 0.f;

    int buf = 0;
    for (int c = c_first; c < nch; c += kTcaWarps, buf ^= 1) {
      if (c + kTcaWarps < nch) {
        issue(c + kTcaWarps, buf ^ 1);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      __syncwarp();
      const int cnt = min(kTcaChunk, s1 - (s0 + c * kTcaChunk));
      const bf16* Ks = wbuf + (size_t)buf * 2 * kTcaChunk * KROW;
      const bf16* Vs = Ks + kTcaChunk * KROW;
      // logits: 4 n-tiles of 8 positions
      float s[4][2];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        s[t][0] = s[t][1] = 0.f;
        const bf16* kr = Ks + (size_t)(t * 8 + (lane & 7)) * KROW + 8 * (lane >> 3);
#pragma unroll
        for (int kk = 0; kk < KSTEPS; kk += 2) {
          uint32_t b0, b1, b2, b3;
          tca::ldsm_x4(kr + kk * 16, b0, b1, b2, b3);
          tca::mma16816(s[t][0], s[t][1], z, qh[kk][0], qh[kk][1], b0, b1);
          tca::mma16816(s[t][0], s[t][1], z, qh[kk + 1][0], qh[kk + 1][1], b2, b3);
          if (SPLIT) {
            tca::mma16816(s[t][0], s[t][1], z, ql[kk][0], ql[kk][1], b0, b1);
            tca::mma16816(s[t][0], s[t][1], z, ql[kk + 1][0], ql[kk + 1][1], b2, b3);
          }
        }
      }
      // online softmax of row h0 over positions t*8 + c2 (+1)
      float cm = -INFINITY;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (t * 8 + c2 >= cnt) s[t][0] = -INFINITY;
        if (t * 8 + c2 + 1 >= cnt) s[t][1] = -INFINITY;
        cm = fmaxf(cm, fmaxf(s[t][0], s[t][1]));
      }
      cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 1));
      cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 2));
      const float mn = fmaxf(mrun, cm);
      const float alpha = mrun == -INFINITY ? 0.f : expf(mrun - mn);
      float ps = 0.f;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        s[t][0] = expf(s[t][0] - mn);
        s[t][1] = expf(s[t][1] - mn);
        ps += s[t][0] + s[t][1];
      }
      ps += __shfl_xor_sync(0xffffffffu, ps, 1);
      ps += __shfl_xor_sync(0xffffffffu, ps, 2);
      lrun = lrun * alpha + ps;
      mrun = mn;
#pragma unroll
      for (int t = 0; t < DT; ++t) {
        o[t][0] *= alpha;
        o[t][1] *= alpha;
      }
      // O += P V: two k-steps of 16 positions
#pragma unroll
      for (int k2 = 0; k2 < 2; ++k2) {
        uint32_t ah0, ah2, al0 = 0, al2 = 0;
        if (SPLIT) {
          tca::split_pack(s[2 * k2][0], s[2 * k2][1], ah0, al0);
          tca::split_pack(s[2 * k2 + 1][0], s[2 * k2 + 1][1], ah2, al2);
        } else {
          ah0 = tca::pack_bf16(s[2 * k2][0], s[2 * k2][1]);
          ah2 = tca::pack_bf16(s[2 * k2 + 1][0], s[2 * k2 + 1][1]);
        }
        // lanes 0-7 / 8-15: positions 16*k2 + 0..7 / 8..15 of dims 8t..; 16-31: dims 8(t+1)..
        const bf16* vr = Vs + (size_t)(k2 * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * KROW + 8 * (lane >> 4);
#pragma unroll
        for (int t = 0; t < DT; t += 2) {
          uint32_t b0, b1, b2, b3;
          tca::ldsm_x4_t(vr + t * 8, b0, b1, b2, b3);
          tca::mma16816(o[t][0], o[t][1], z, ah0, ah2, b0, b1);
          tca::mma16816(o[t + 1][0], o[t + 1][1], z, ah0, ah2, b2, b3);
          if (SPLIT) {
            tca::mma16816(o[t][0], o[t][1], z, al0, al2, b0, b1);
            tca::mma16816(o[t + 1][0], o[t + 1][1], z, al0, al2, b2, b3);
          }
        }
      }
      __syncwarp();   // the buffer is refilled by the issue two chunks on
    }
    // combine the four warps (the K/V buffers are free once all are done)
    __syncthreads();
    if ((lane & 3) == 0) {
      mw[warp * 8 + h0] = mrun;
      lw[warp * 8 + h0] = lrun;
    }
#pragma unroll
    for (int t = 0; t < DT; ++t) {
      float* d = ow + ((size_t)warp * 8 + h0) * HD + t * 8 + c2;
      d[0] = o[t][0];
      d[1] = o[t][1];
    }
    __syncthreads();
    const size_t obase = (size_t)j * nq * HD + (size_t)g * G * HD;
    for (int x = tid; x < G * HD; x += kTcaThreads) {
      const int h = x / HD, e = x - h * HD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kTcaWarps; ++w) M = fmaxf(M, mw[w * 8 + h]);
      float L = 0.f, O = 0.f;
#pragma unroll
      for (int w = 0; w < kTcaWarps; ++w) {
        const float mv = mw[w * 8 + h];
        const float f = mv == -INFINITY ? 0.f : expf(mv - M);
        L += lw[w * 8 + h] * f;
        O += ow[((size_t)w * 8 + h) * HD + e] * f;
      }
      if (nsp == 1) {
        store_out(A.out, A.out_lo, obase + x, O / L);
      } else {
        const size_t slot = ((size_t)j * nq + g * G + h) * A.max_spans + sp;
        __stcg(A.part_acc + slot * HD + e, O);
        if (e == 0) {
          __stcg(A.part_m + slot, M);
          __stcg(A.part_l + slot, L);
        }
      }
    }
    if (nsp > 1) {
      __syncthreads();
      if (tid == 0) {
        __threadfence();
        const int old = atomicAdd(&A.ctr[j * nkv + g], 1);
        *last_s_p = (old == nsp - 1);
        if (*last_s_p) A.ctr[j * nkv + g] = 0;
        __threadfence();
      }
      __syncthreads();
      if (*last_s_p) attn_span_merge<bf16, HD, kTcaThreads>(A, j, g, nsp, obase, tid);
    }
    __syncthreads();
  }
  if (!waited) {
    pdl_wait();
    pdl_trigger();
  }
}

}  // namespace buddy

// Decode attention on the tensor cores (bf16 caches, head dim 64 or 128, at
// most 8 query heads per KV head), Eq. 9 for every active row and KV head.
//
// Work decomposition: the (row j, KV head g) streams of positions 0..len[i]
// are laid end to end (row-major, heads inside a row) and every warp of the
// grid takes an equal contiguous share of that sequence (a multiple of the
// chunk, at least two chunks).  A share may end in the middle of a stream and
// cover several short ones; the piece of a stream that one warp holds is a
// span.  A stream held by one warp is written out directly; otherwise every
// warp writes its span's partial (running max, sum of exponentials,
// unnormalised output), and the warp that completes the stream last (an
// arrival counter per stream) merges the partials in span order
// (deterministic), kTcaWarpMerge spans' loads at a time.  Because warps never
// wait for each other, each streams its share without a break: the copies of
// the next span are in flight while the current one finishes (or merges), and
// no second kernel is needed.
//
// Inside a share a warp walks chunks of up to kTcaChunk positions (never
// crossing a stream end):
//
//   * K and V rows of the chunk are copied with 16-byte cp.async into one of
//     the warp's kTcaStages buffers (rows padded by 16 bytes: ldmatrix
//     conflict-free); kTcaStages - 1 chunks are in flight while one is used;
//   * logits, transposed: S^T = K Q^T with mma.sync m16n8k16 (bf16 in, fp32
//     accumulate): 16 positions are the rows of A (K rows through ldmatrix),
//     the query heads the 8 columns of B (heads >= G are zero);
//   * online softmax per head (a column) on the accumulator fragments, in
//     base 2 (the queries carry log2(e) / sqrt(d_h));
//   * O^T += V^T P^T: 16 channels are the rows of A (V through
//     ldmatrix.trans), the probabilities, transposed in registers
//     (movmatrix), the B operand.
//
// With SPLIT (the first block, which feeds the router) the scaled queries and
// the probabilities are each given as bf16 hi + lo and every product is issued
// for both terms, so the contractions carry ~16 mantissa bits; otherwise one
// bf16 term each.
#pragma once

#include <cuda_runtime.h>

#include "attn_common.cuh"
#include "common.cuh"
#include "ptx.cuh"

namespace buddy {

constexpr int kTcaChunk = 32;     // positions per warp chunk (16 or 32)
constexpr int kTcaWarps = 4;
constexpr int kTcaThreads = 32 * kTcaWarps;
constexpr int kTcaStages = 3;     // chunk buffers per warp (kTcaStages - 1 in flight)
constexpr int kTcaMinShare = 2 * kTcaChunk;   // positions of a warp's share, at least
constexpr int kTcaWarpMerge = 4;              // span partials loaded at a time by the merging warp

template <int HD>
__host__ __device__ constexpr size_t attn_tc_smem_fixed() {
  // per warp: kTcaStages buffers of K and V rows, each row padded by 8 bf16
  return (size_t)kTcaWarps * kTcaStages * 2 * kTcaChunk * (HD + 8) * 2;
}
constexpr int kTcaSmemLimit = 226 * 1024;   // dynamic shared memory of one CTA (227 KiB less static)
inline size_t attn_tc_smem_bytes(int hd, int max_rows) {
  const size_t fixed = hd == 128 ? attn_tc_smem_fixed<128>() : attn_tc_smem_fixed<64>();
  return fixed + (size_t)(max_rows + 1) * 4 + 8 + (size_t)max_rows * 16;
}
// Spans one stream of at most max_pos positions can be cut into: shares are at
// least kTcaMinShare positions, and the first and last may be partial.
inline int attn_tc_max_spans(int max_pos) { return (max_pos + kTcaMinShare - 1) / kTcaMinShare + 1; }

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
// D (16x8 fp32) += A (16x16 bf16) * B (16x8 bf16)
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// transpose of an 8x8 b16 matrix held one 32-bit pair per thread
__device__ __forceinline__ uint32_t movt(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// 2^x (hardware approximation, relative error ~2^-22; 2^-inf = 0)
__device__ __forceinline__ float exp2a(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

}  // namespace tca

// Merge of a (row j, KV head g)'s nsp span partials by one warp: lane ->
// (head, four channels) per round of 32 lanes.  For two rounds at a time the
// partials (output, max and sum) of kTcaWarpMerge spans are loaded at once and
// folded into a running max M, sum L and output O in span order (a group
// raising M rescales what came before by 2^(M_old - M_new)); the result is
// O / L, i.e. sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s.
template <int HD>
__device__ __forceinline__ void attn_tc_warp_merge(const AttnArgs<bf16>& A, int j, int g, int nsp, size_t obase,
                                                   int lane) {
  constexpr int Q = HD / 4;      // float4 outputs per head
  constexpr int HPR = 32 / Q;    // heads per round (1 or 2)
  constexpr int NS = kTcaWarpMerge;
  const int G = A.nq / A.nkv, ms = A.max_spans;
  const size_t hb0 = ((size_t)j * A.nq + (size_t)g * G) * ms;
  const int hsub = lane / Q, e0 = (lane % Q) * 4;
  for (int r0 = 0; r0 * HPR < G; r0 += 2) {
    float M[2] = {-INFINITY, -INFINITY}, L[2] = {0.f, 0.f};
    float4 acc[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
    for (int s0 = 0; s0 < nsp; s0 += NS) {
      float4 v[2][NS];
      float mv[2][NS], lv[2][NS];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int h = (r0 + u) * HPR + hsub;
#pragma unroll
        for (int s = 0; s < NS; ++s) {
          if (h < G && s0 + s < nsp) {
            const size_t slot = hb0 + (size_t)h * ms + s0 + s;
            v[u][s] = __ldcg(reinterpret_cast<const float4*>(A.part_acc + slot * HD + e0));
            mv[u][s] = __ldcg(A.part_m + slot);
            lv[u][s] = __ldcg(A.part_l + slot);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int h = (r0 + u) * HPR + hsub;
        if (h >= G) continue;
        float mn = M[u];
#pragma unroll
        for (int s = 0; s < NS; ++s)
          if (s0 + s < nsp) mn = fmaxf(mn, mv[u][s]);
        // span maxima are finite, so mn is; 2^(-inf) = 0 on the first group
        const float sc = tca::exp2a(M[u] - mn);
        M[u] = mn;
        L[u] *= sc;
        acc[u].x *= sc;
        acc[u].y *= sc;
        acc[u].z *= sc;
        acc[u].w *= sc;
#pragma unroll
        for (int s = 0; s < NS; ++s) {
          if (s0 + s < nsp) {
            const float w = tca::exp2a(mv[u][s] - mn);
            L[u] += w * lv[u][s];
            acc[u].x += w * v[u][s].x;
            acc[u].y += w * v[u][s].y;
            acc[u].z += w * v[u][s].z;
            acc[u].w += w * v[u][s].w;
          }
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int h = (r0 + u) * HPR + hsub;
      if (h >= G) continue;
      const float inv = 1.f / L[u];
      const size_t o = obase + (size_t)h * HD + e0;
      store_out(A.out, A.out_lo, o + 0, acc[u].x * inv);
      store_out(A.out, A.out_lo, o + 1, acc[u].y * inv);
      store_out(A.out, A.out_lo, o + 2, acc[u].z * inv);
      store_out(A.out, A.out_lo, o + 3, acc[u].w * inv);
    }
  }
}

// Position in the sequence of streams: row j (index into the active rows), KV
// head g, position p of that stream (np = the stream's length).
struct TcaCursor {
  int j, g, p, np;
};

// Processes warp `gw` of `nw` warps' share of one layer's attention.  Smem:
// per-warp K/V buffers, then the row prefix (stream starts of each row, in
// positions) and the rows' cache offsets, lengths and head strides, written by
// warp 0 of every CTA before the CTA-wide barrier.
template <int HD, bool SPLIT>
__device__ __forceinline__ void attn_tc_run(const AttnArgs<bf16>& A, int cta, int ncta, uint8_t* smem, int* sc,
                                            bool pdl) {
  static_assert(HD == 64 || HD == 128, "HD");
  static_assert(kTcaChunk == 16 || kTcaChunk == 32, "chunk");
  constexpr int CH = kTcaChunk, NST = kTcaStages;
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
  bf16* wbuf = reinterpret_cast<bf16*>(smem) + (size_t)warp * NST * 2 * CH * KROW;   // this warp's buffers
  int* pref = reinterpret_cast<int*>(smem + attn_tc_smem_fixed<HD>());
  int64_t* rbase = reinterpret_cast<int64_t*>((reinterpret_cast<uintptr_t>(pref + m + 1) + 7) & ~uintptr_t(7));
  int* rnp = reinterpret_cast<int*>(rbase + m);
  int* rhs = rnp + m;

  // streams per row (nkv of length len + 1) and their prefix; the share
  if (warp == 0) {
    int carry = 0;
    for (int b = 0; b < m; b += 32) {
      const int j = b + lane;
      int x = 0;
      if (j < m) {
        const int i = rows ? rows[j] : j;
        const int np = A.len[i] + 1;
        rnp[j] = np;
        rbase[j] = A.seq_off[i] * nkv * HD;
        rhs[j] = A.cap[i] * HD;
        x = np * nkv;
      }
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (j < m) pref[j + 1] = carry + x;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) {
      pref[0] = 0;
      const int nw = ncta * kTcaWarps;
      const int even = (carry + nw - 1) / nw;
      sc[0] = max(kTcaMinShare, (even + CH - 1) / CH * CH);
    }
  }
  __syncthreads();
  const int share = sc[0];
  const int total = pref[m];
  const int gw = cta * kTcaWarps + warp;
  const long long a0 = (long long)gw * share;
  if (a0 >= total) {   // nothing for this warp
    if (pdl) {
      pdl_wait();
      pdl_trigger();
    }
    return;
  }
  const int a = (int)a0, b = min(total, a + share);

  // cursor at flattened position x (binary search of the row prefix)
  auto seek = [&](int x) {
    int lo = 0, hi = m;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pref[mid] <= x) lo = mid;
      else hi = mid;
    }
    TcaCursor c;
    c.j = lo;
    c.np = rnp[lo];
    const int off = x - pref[lo];
    c.g = off / c.np;
    c.p = off - c.g * c.np;
    return c;
  };
  // positions of the chunk at cursor c (flattened position x)
  auto chunk_len = [&](const TcaCursor& c, int x) { return min(CH, min(c.np - c.p, b - x)); };
  // advance past a chunk of n positions (never beyond the stream end)
  auto advance = [&](TcaCursor& c, int n) {
    c.p += n;
    if (c.p == c.np) {
      c.p = 0;
      if (++c.g == nkv) {
        c.g = 0;
        if (++c.j < m) c.np = rnp[c.j];
      }
    }
  };
  auto issue = [&](const TcaCursor& c, int cnt, int buf) {
    const int64_t kvo = rbase[c.j] + (int64_t)c.g * rhs[c.j] + (int64_t)c.p * HD;
    bf16* Kd = wbuf + (size_t)buf * 2 * CH * KROW;
    bf16* Vd = Kd + CH * KROW;
    // lane -> (row lane / V16 + RPI * i, 16-byte piece lane % V16)
    constexpr int RPI = 32 / V16;
    const int pl = lane / V16, sl = lane % V16;
    const bf16* ks = A.Kc + kvo + pl * HD + sl * 8;
    const bf16* vs = A.Vc + kvo + pl * HD + sl * 8;
    const int so = pl * KROW + sl * 8;
#pragma unroll 4
    for (int r = 0; r + pl < cnt; r += RPI) {
      cp_async16(Kd + so + r * KROW, ks + (size_t)r * HD);
      cp_async16(Vd + so + r * KROW, vs + (size_t)r * HD);
    }
    // rows past the chunk end: zero V (their probabilities are 0, and 0 times
    // stale shared memory could be NaN); K is masked on the logits
    for (int x = cnt * V16 + lane; x < CH * V16; x += 32) {
      const int r = x / V16, q = x - r * V16;
      *reinterpret_cast<uint4*>(Vd + r * KROW + q * 8) = make_uint4(0u, 0u, 0u, 0u);
    }
  };

  // prologue: kTcaStages - 1 chunks in flight (one commit group each, empty
  // past the share); chunks without the new token (the last position of a
  // stream, written by the preceding kernel) may be copied before the wait
  TcaCursor ci = seek(a);
  int xi = a;
  int k0 = 0;
  if (pdl) {
    for (; k0 < NST - 1 && xi < b; ++k0) {
      const int cnt = chunk_len(ci, xi);
      if (ci.p + cnt == ci.np) break;
      issue(ci, cnt, k0);
      cp_async_commit();
      advance(ci, cnt);
      xi += cnt;
    }
    pdl_wait();
    pdl_trigger();
  }
  for (int k = k0; k < NST - 1; ++k) {
    if (xi < b) {
      const int cnt = chunk_len(ci, xi);
      issue(ci, cnt, k);
      advance(ci, cnt);
      xi += cnt;
    }
    cp_async_commit();
  }

  const float scale = 1.4426950408889634f * rsqrtf((float)HD);   // log2(e) / sqrt(d_h)
  const int h0 = lane >> 2, c2 = (lane & 3) * 2;   // fragment row (head) and column pair
  TcaCursor cc = seek(a);
  int xc = a;
  uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
  float mrun[2], lrun[2];   // heads c2, c2 + 1
  float o[DT / 2][4];       // O^T: channels 16 * t + lane / 4 (+8) x heads c2, c2 + 1
  for (int k = 0; xc < b; ++k) {
    if (xi < b) {
      const int cnt = chunk_len(ci, xi);
      issue(ci, cnt, (k + NST - 1) % NST);
      advance(ci, cnt);
      xi += cnt;
    }
    cp_async_commit();
    const int cnt = chunk_len(cc, xc);
    if (xc == a || cc.p == 0) {
      // a new span: query fragments as the B operand (column = head h0 < G,
      // rows = dims), scaled by log2(e) / sqrt(d_h), and a fresh running state
      const float* qj = A.q + ((size_t)cc.j * nq + (size_t)cc.g * G + h0) * HD;
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        float x0 = 0.f, x1 = 0.f, x2 = 0.f, x3 = 0.f;
        if (h0 < G) {
          const float2 u = *reinterpret_cast<const float2*>(qj + kk * 16 + c2);
          const float2 v = *reinterpret_cast<const float2*>(qj + kk * 16 + 8 + c2);
          x0 = u.x * scale; x1 = u.y * scale; x2 = v.x * scale; x3 = v.y * scale;
        }
        if (SPLIT) {
          tca::split_pack(x0, x1, qh[kk][0], ql[kk][0]);
          tca::split_pack(x2, x3, qh[kk][1], ql[kk][1]);
        } else {
          qh[kk][0] = tca::pack_bf16(x0, x1);
          qh[kk][1] = tca::pack_bf16(x2, x3);
        }
      }
      mrun[0] = mrun[1] = -INFINITY;
      lrun[0] = lrun[1] = 0.f;
#pragma unroll
      for (int t = 0; t < DT / 2; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
    }
    cp_async_wait<NST - 1>();
    __syncwarp();
    const bf16* Ks = wbuf + (size_t)(k % NST) * 2 * CH * KROW;
    const bf16* Vs = Ks + CH * KROW;
    // S^T for MT tiles of 16 positions: two accumulators per tile (even and
    // odd k-steps) for independent MMA chains
    constexpr int MT = CH / 16;
    float sv[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
      // lanes 0-7 / 8-15: positions 16*mt + 0..7 / 8..15 of dims 16kk + 0..7;
      // lanes 16-31: the same positions, dims 16kk + 8..15
      const bf16* kr = Ks + (size_t)(mt * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * KROW + 8 * (lane >> 4);
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t a0, a1, a2, a3;
        tca::ldsm_x4(kr + kk * 16, a0, a1, a2, a3);
        tca::mma16816(acc[kk & 1], a0, a1, a2, a3, qh[kk][0], qh[kk][1]);
        if (SPLIT) tca::mma16816(acc[kk & 1], a0, a1, a2, a3, ql[kk][0], ql[kk][1]);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) sv[mt][i] = acc[0][i] + acc[1][i];
    }
    // online softmax per head: this lane holds positions 16*mt + lane/4 (+8)
    // of heads c2 (elements 0, 2) and c2 + 1 (elements 1, 3)
    float cm[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      const int p0 = mt * 16 + h0;
      if (p0 >= cnt) sv[mt][0] = sv[mt][1] = -INFINITY;
      if (p0 + 8 >= cnt) sv[mt][2] = sv[mt][3] = -INFINITY;
      cm[0] = fmaxf(cm[0], fmaxf(sv[mt][0], sv[mt][2]));
      cm[1] = fmaxf(cm[1], fmaxf(sv[mt][1], sv[mt][3]));
    }
    float alpha[2], ps[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) cm[e] = fmaxf(cm[e], __shfl_xor_sync(0xffffffffu, cm[e], off));
      const float mn = fmaxf(mrun[e], cm[e]);
      alpha[e] = tca::exp2a(mrun[e] - mn);   // 0 while mrun is -inf
      mrun[e] = mn;
      ps[e] = 0.f;
    }
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        sv[mt][i] = tca::exp2a(sv[mt][i] - mrun[i & 1]);
        ps[i & 1] += sv[mt][i];
      }
    }
#pragma unroll
    for (int e = 0; e < 2; ++e) {
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) ps[e] += __shfl_xor_sync(0xffffffffu, ps[e], off);
      lrun[e] = lrun[e] * alpha[e] + ps[e];
    }
#pragma unroll
    for (int t = 0; t < DT / 2; ++t) {
      o[t][0] *= alpha[0];
      o[t][1] *= alpha[1];
      o[t][2] *= alpha[0];
      o[t][3] *= alpha[1];
    }
    // O^T += V^T P^T, one k-step per tile of 16 positions
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      // P^T as B: transpose of the (positions x heads) fragments
      uint32_t bh0, bh1, bl0 = 0, bl1 = 0;
      if (SPLIT) {
        uint32_t x0, y0, x1, y1;
        tca::split_pack(sv[mt][0], sv[mt][1], x0, y0);
        tca::split_pack(sv[mt][2], sv[mt][3], x1, y1);
        bh0 = tca::movt(x0);
        bh1 = tca::movt(x1);
        bl0 = tca::movt(y0);
        bl1 = tca::movt(y1);
      } else {
        bh0 = tca::movt(tca::pack_bf16(sv[mt][0], sv[mt][1]));
        bh1 = tca::movt(tca::pack_bf16(sv[mt][2], sv[mt][3]));
      }
      // ldmatrix.trans groups: lanes 0-7 / 8-15 / 16-23 / 24-31 address
      // positions 0..7 / 0..7 / 8..15 / 8..15 at channels +0 / +8 / +0 / +8
      const bf16* vr = Vs + (size_t)(mt * 16 + (lane & 7) + 8 * (lane >> 4)) * KROW + 8 * ((lane >> 3) & 1);
#pragma unroll
      for (int t = 0; t < DT / 2; ++t) {
        uint32_t a0, a1, a2, a3;
        tca::ldsm_x4_t(vr + t * 16, a0, a1, a2, a3);
        tca::mma16816(o[t], a0, a1, a2, a3, bh0, bh1);
        if (SPLIT) tca::mma16816(o[t], a0, a1, a2, a3, bl0, bl1);
      }
    }
    __syncwarp();   // the buffer is refilled by the next iteration's issue

    const TcaCursor cs = cc;   // the span this chunk belongs to
    advance(cc, cnt);
    xc += cnt;
    if (cs.p + cnt == cs.np || xc == b) {
      // end of the span: its stream covers flattened [S0, S0 + np), cut by the
      // shares into spans first .. last (this warp's is gw - first)
      const int S0 = pref[cs.j] + cs.g * cs.np;
      const int first = S0 / share, nsp = (S0 + cs.np - 1) / share - first + 1;
      const size_t obase = ((size_t)cs.j * nq + (size_t)cs.g * G) * HD;
      // this lane: heads c2 + e (e = 0, 1), channels 16 t + h0 (+ 8)
      if (nsp == 1) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          if (c2 + e < G) {
            const float inv = 1.f / lrun[e];
            const size_t ob = obase + (size_t)(c2 + e) * HD + h0;
#pragma unroll
            for (int t = 0; t < DT / 2; ++t) {
              store_out(A.out, A.out_lo, ob + 16 * t, o[t][e] * inv);
              store_out(A.out, A.out_lo, ob + 16 * t + 8, o[t][2 + e] * inv);
            }
          }
        }
      } else {   // a partial, merged by the warp that completes the stream
        const int sp = gw - first;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          if (c2 + e < G) {
            const size_t slot = ((size_t)cs.j * nq + (size_t)cs.g * G + c2 + e) * A.max_spans + sp;
            float* pa = A.part_acc + slot * HD + h0;
#pragma unroll
            for (int t = 0; t < DT / 2; ++t) {
              __stcg(pa + 16 * t, o[t][e]);
              __stcg(pa + 16 * t + 8, o[t][2 + e]);
            }
            if (h0 == 0) {
              __stcg(A.part_m + slot, mrun[e]);
              __stcg(A.part_l + slot, lrun[e]);
            }
          }
        }
        // the partial is visible before the arrival is counted; the warp
        // that completes the stream merges (and re-arms the counter)
        __syncwarp();
        int last = 0;
        if (lane == 0) {
          int32_t* ctr = A.ctr + cs.j * nkv + cs.g;
          const int old = ptx::atom_add_acq_rel(ctr, 1);
          last = old == nsp - 1;
          if (last) *ctr = 0;   // re-armed for a later launch
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        __syncwarp();
        if (last) attn_tc_warp_merge<HD>(A, cs.j, cs.g, nsp, obase, lane);
      }
    }
  }
}

}  // namespace buddy

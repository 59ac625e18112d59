// Causal attention of a prefill block (App. E, Eq. 9 applied to every prompt
// token): the query of prompt token t of sequence i, at cache position
// c0 + t of the block's cache (c0 = the positions it held before the
// prompt), attends to cache positions 0 .. c0 + t.
//
// A CTA takes one work item: 64 query tokens of one sequence and one query
// head (4 warps x 16 tokens).  It walks the key/value positions of the KV
// head in tiles of 64, copied with 16-byte cp.async into two shared-memory
// buffers (one tile in flight while the other is used; rows padded by 16
// bytes so that ldmatrix is conflict-free).  Per tile and warp:
//   S = Q K^T      mma.sync m16n8k16, the 16 tokens as A (from registers),
//                  K rows through ldmatrix as B; 8 position tiles x HD/16
//                  k-steps;
//   online softmax per token in base 2 (queries pre-scaled by
//                  log2(e) / sqrt(d_h)), causal and range masks;
//   O += P V       the probabilities re-packed from the S fragments as A,
//                  V through ldmatrix.trans as B; HD/8 channel tiles x 4
//                  k-steps.
// With SPLIT (the blocks that feed the router) the queries and the
// probabilities are each given as bf16 hi + lo and every product is issued
// for both terms.
#include <cuda_runtime.h>

#include "attn_tc.cuh"
#include "common.cuh"
#include "internal.h"

namespace buddy {

constexpr int kPfaThreads = 128;
constexpr int kPfaRows = 64;    // query tokens per work item
constexpr int kPfaKeys = 64;    // key positions per tile

template <int HD>
__host__ __device__ constexpr size_t attn_pf_smem() {
  return (size_t)2 * 2 * kPfaKeys * (HD + 8) * sizeof(bf16);   // 2 buffers x (K, V)
}

struct PfaArgs {
  const int4* items;        // (sequence, query head, first compact row, first prompt token)
  const int32_t* n_tok;     // sequence -> prompt tokens
  const int32_t* base;      // sequence -> positions the layer's cache held before the prompt
  const float* q;           // [m, nq * hd] compact rows
  const int64_t* seq_off;
  const int32_t* cap;
  const bf16* Kc;
  const bf16* Vc;
  bf16* out;                // [m, nq * hd]
  bf16* out_lo;
  int nq, nkv;
  const int32_t* status;
};

template <int HD, bool SPLIT>
__global__ void __launch_bounds__(kPfaThreads) attn_pf_kernel(PfaArgs A) {
  extern __shared__ __align__(16) uint8_t smraw[];
  constexpr int KROW = HD + 8;
  constexpr int KSTEPS = HD / 16;
  constexpr int NT = kPfaKeys / 8;    // position tiles of the logits
  constexpr int DT = HD / 8;          // channel tiles of the output
  constexpr int V16 = HD / 8;         // 16-byte pieces per row
  if (call_aborted(A.status)) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int4 it = A.items[blockIdx.x];
  const int seq = it.x, h = it.y, j0 = it.z, t0 = it.w;
  const int G = A.nq / A.nkv, g = h / G;
  const int ntok = A.n_tok[seq];
  const int c0 = A.base[seq];
  const int nrow = min(kPfaRows, ntok - t0);
  const int kmax = c0 + t0 + nrow;    // positions the last query of the item sees
  const int64_t kvbase = (A.seq_off[seq] * A.nkv + (int64_t)g * A.cap[seq]) * HD;
  bf16* sK[2];
  bf16* sV[2];
  sK[0] = reinterpret_cast<bf16*>(smraw);
  sV[0] = sK[0] + kPfaKeys * KROW;
  sK[1] = sV[0] + kPfaKeys * KROW;
  sV[1] = sK[1] + kPfaKeys * KROW;

  auto issue = [&](int kt, int buf) {
    const int p0 = kt * kPfaKeys;
    const int cnt = min(kPfaKeys, kmax - p0);
    for (int x = tid; x < kPfaKeys * V16; x += kPfaThreads) {
      const int r = x / V16, q16 = x - r * V16;
      bf16* kd = sK[buf] + r * KROW + q16 * 8;
      bf16* vd = sV[buf] + r * KROW + q16 * 8;
      if (r < cnt) {
        const size_t off = (size_t)(kvbase + (int64_t)(p0 + r) * HD + q16 * 8);
        cp_async16(kd, A.Kc + off);
        cp_async16(vd, A.Vc + off);
      } else {   // rows past the range: zero (their probabilities are 0; 0 * stale could be NaN)
        *reinterpret_cast<uint4*>(kd) = make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(vd) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
  };

  const int ntiles = (kmax + kPfaKeys - 1) / kPfaKeys;
  issue(0, 0);
  cp_async_commit();

  // queries of this warp's 16 tokens as A fragments: row r = lane / 4 (+ 8),
  // columns 2 (lane % 4) (+ 1) (+ 8) of each k-step; pre-scaled
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);
  const int gr = lane >> 2, tc = (lane & 3) * 2;
  const int rA = warp * 16 + gr, rB = rA + 8;          // rows within the item
  const bool vA = rA < nrow, vB = rB < nrow;
  const float* qA = A.q + ((size_t)(j0 + rA) * A.nq + h) * HD;
  const float* qB = A.q + ((size_t)(j0 + rB) * A.nq + h) * HD;
  uint32_t qh[KSTEPS][4], ql[KSTEPS][4];
#pragma unroll
  for (int kk = 0; kk < KSTEPS; ++kk) {
    float2 a0 = vA ? *reinterpret_cast<const float2*>(qA + kk * 16 + tc) : make_float2(0.f, 0.f);
    float2 a1 = vB ? *reinterpret_cast<const float2*>(qB + kk * 16 + tc) : make_float2(0.f, 0.f);
    float2 a2 = vA ? *reinterpret_cast<const float2*>(qA + kk * 16 + 8 + tc) : make_float2(0.f, 0.f);
    float2 a3 = vB ? *reinterpret_cast<const float2*>(qB + kk * 16 + 8 + tc) : make_float2(0.f, 0.f);
    const float2 f[4] = {a0, a1, a2, a3};
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      if (SPLIT) tca::split_pack(f[r].x * scale, f[r].y * scale, qh[kk][r], ql[kk][r]);
      else qh[kk][r] = tca::pack_bf16(f[r].x * scale, f[r].y * scale);
    }
  }
  const int qposA = c0 + t0 + rA, qposB = c0 + t0 + rB;   // cache positions of the two rows
  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  float o[DT][4];
#pragma unroll
  for (int t = 0; t < DT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;

  for (int kt = 0; kt < ntiles; ++kt) {
    const int buf = kt & 1;
    if (kt + 1 < ntiles) issue(kt + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const bf16* Ks = sK[buf];
    const bf16* Vs = sV[buf];
    const int p0 = kt * kPfaKeys;
    // ---- S = Q K^T: 16 tokens x 64 positions
    float s[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int np = 0; np < NT; np += 2) {
      // ldmatrix x4: positions 8 np.. / 8 (np + 1).., dims +0 / +8 of a k-step
      const int m4 = lane >> 3, r8 = lane & 7;
      const bf16* kr = Ks + (size_t)(8 * np + 8 * (m4 >> 1) + r8) * KROW + 8 * (m4 & 1);
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t b0, b1, b2, b3;
        tca::ldsm_x4(kr + kk * 16, b0, b1, b2, b3);
        tca::mma16816(s[np], qh[kk][0], qh[kk][1], qh[kk][2], qh[kk][3], b0, b1);
        tca::mma16816(s[np + 1], qh[kk][0], qh[kk][1], qh[kk][2], qh[kk][3], b2, b3);
        if (SPLIT) {
          tca::mma16816(s[np], ql[kk][0], ql[kk][1], ql[kk][2], ql[kk][3], b0, b1);
          tca::mma16816(s[np + 1], ql[kk][0], ql[kk][1], ql[kk][2], ql[kk][3], b2, b3);
        }
      }
    }
    // ---- masks and online softmax (rows A = gr, B = gr + 8)
    float cmA = -INFINITY, cmB = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int pp = p0 + nt * 8 + tc;
      if (pp > qposA) s[nt][0] = -INFINITY;
      if (pp + 1 > qposA) s[nt][1] = -INFINITY;
      if (pp > qposB) s[nt][2] = -INFINITY;
      if (pp + 1 > qposB) s[nt][3] = -INFINITY;
      cmA = fmaxf(cmA, fmaxf(s[nt][0], s[nt][1]));
      cmB = fmaxf(cmB, fmaxf(s[nt][2], s[nt][3]));
    }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      cmA = fmaxf(cmA, __shfl_xor_sync(0xffffffffu, cmA, off));
      cmB = fmaxf(cmB, __shfl_xor_sync(0xffffffffu, cmB, off));
    }
    // position 0 of tile 0 is visible to every row, so the running max is
    // finite from the first tile on
    const float nmA = fmaxf(mA, cmA), nmB = fmaxf(mB, cmB);
    const float alA = tca::exp2a(mA - nmA), alB = tca::exp2a(mB - nmB);
    mA = nmA;
    mB = nmB;
    float psA = 0.f, psB = 0.f;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      s[nt][0] = tca::exp2a(s[nt][0] - mA);
      s[nt][1] = tca::exp2a(s[nt][1] - mA);
      s[nt][2] = tca::exp2a(s[nt][2] - mB);
      s[nt][3] = tca::exp2a(s[nt][3] - mB);
      psA += s[nt][0] + s[nt][1];
      psB += s[nt][2] + s[nt][3];
    }
    lA = lA * alA + psA;   // per-thread partial sums; the quad is reduced at the end
    lB = lB * alB + psB;
#pragma unroll
    for (int t = 0; t < DT; ++t) {
      o[t][0] *= alA;
      o[t][1] *= alA;
      o[t][2] *= alB;
      o[t][3] *= alB;
    }
    // ---- O += P V: k-steps of 16 positions (two position tiles)
#pragma unroll
    for (int kk = 0; kk < NT / 2; ++kk) {
      uint32_t ah[4], al[4] = {0u, 0u, 0u, 0u};
      if (SPLIT) {
        tca::split_pack(s[2 * kk][0], s[2 * kk][1], ah[0], al[0]);
        tca::split_pack(s[2 * kk][2], s[2 * kk][3], ah[1], al[1]);
        tca::split_pack(s[2 * kk + 1][0], s[2 * kk + 1][1], ah[2], al[2]);
        tca::split_pack(s[2 * kk + 1][2], s[2 * kk + 1][3], ah[3], al[3]);
      } else {
        ah[0] = tca::pack_bf16(s[2 * kk][0], s[2 * kk][1]);
        ah[1] = tca::pack_bf16(s[2 * kk][2], s[2 * kk][3]);
        ah[2] = tca::pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
        ah[3] = tca::pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
      }
      // ldmatrix.trans x4: positions 16 kk + 0..7 / + 8..15, channels +0 / +8
      const int m4 = lane >> 3, r8 = lane & 7;
      const bf16* vr = Vs + (size_t)(16 * kk + 8 * (m4 & 1) + r8) * KROW + 8 * (m4 >> 1);
#pragma unroll
      for (int t = 0; t < DT; t += 2) {
        uint32_t b0, b1, b2, b3;
        tca::ldsm_x4_t(vr + t * 8, b0, b1, b2, b3);
        tca::mma16816(o[t], ah[0], ah[1], ah[2], ah[3], b0, b1);
        tca::mma16816(o[t + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
        if (SPLIT) {
          tca::mma16816(o[t], al[0], al[1], al[2], al[3], b0, b1);
          tca::mma16816(o[t + 1], al[0], al[1], al[2], al[3], b2, b3);
        }
      }
    }
    __syncthreads();   // the buffer is refilled by the next iteration's issue
  }
  cp_async_wait<0>();

#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    lA += __shfl_xor_sync(0xffffffffu, lA, off);
    lB += __shfl_xor_sync(0xffffffffu, lB, off);
  }
  const float iA = 1.f / lA, iB = 1.f / lB;
  const size_t qd = (size_t)A.nq * HD;
#pragma unroll
  for (int t = 0; t < DT; ++t) {
    const int ch = h * HD + t * 8 + tc;
    if (vA) {
      store_out(A.out, A.out_lo, (size_t)(j0 + rA) * qd + ch, o[t][0] * iA);
      store_out(A.out, A.out_lo, (size_t)(j0 + rA) * qd + ch + 1, o[t][1] * iA);
    }
    if (vB) {
      store_out(A.out, A.out_lo, (size_t)(j0 + rB) * qd + ch, o[t][2] * iB);
      store_out(A.out, A.out_lo, (size_t)(j0 + rB) * qd + ch + 1, o[t][3] * iB);
    }
  }
}

void launch_attention_pf(const Ctx& c, int n_items, const int4* items, const int32_t* n_tok, const int32_t* base,
                         const buddy_kv_state& kv, int layer, const float* q, void* out, void* out_lo,
                         cudaStream_t s) {
  PfaArgs A{items, n_tok, base, q, kv.seq_off, kv.cap, (const bf16*)kv.k_cache[layer],
            (const bf16*)kv.v_cache[layer], (bf16*)out, (bf16*)out_lo, c.nq, c.nkv, c.status};
  if (c.hd == 128) {
    const size_t smem = attn_pf_smem<128>();
    if (out_lo) {
      cudaFuncSetAttribute(attn_pf_kernel<128, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      attn_pf_kernel<128, true><<<n_items, kPfaThreads, smem, s>>>(A);
    } else {
      cudaFuncSetAttribute(attn_pf_kernel<128, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      attn_pf_kernel<128, false><<<n_items, kPfaThreads, smem, s>>>(A);
    }
  } else {
    const size_t smem = attn_pf_smem<64>();
    if (out_lo) {
      cudaFuncSetAttribute(attn_pf_kernel<64, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      attn_pf_kernel<64, true><<<n_items, kPfaThreads, smem, s>>>(A);
    } else {
      cudaFuncSetAttribute(attn_pf_kernel<64, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      attn_pf_kernel<64, false><<<n_items, kPfaThreads, smem, s>>>(A);
    }
  }
}

}  // namespace buddy

// CUDA-core decode attention work loop, shared by the fp32 attention kernel
// and the per-layer persistent kernel (see attention.cu for the algorithm),
// and the span merge used by both attention loops.
#pragma once

#include <cuda_runtime.h>

#include <algorithm>

#include "common.cuh"

namespace buddy {

constexpr int kChunk = 64;
constexpr int kAttnThreads = 256;   // the attention kernel's CTA (the per-layer kernel uses 128)
constexpr int kMaxSpan = 1024;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <typename T>
__device__ __forceinline__ void load8s(const T* p, float* o);
template <>
__device__ __forceinline__ void load8s<bf16>(const bf16* p, float* o) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[2 * i] = __uint_as_float(w[i] << 16);
    o[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}
template <>
__device__ __forceinline__ void load8s<float>(const float* p, float* o) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
  o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}

// Output in the GEMM input type; with `lo` also the remainder term.
template <typename T>
__device__ __forceinline__ void store_out(T* out, T* lo, size_t i, float v) {
  const T hi = from_f<T>(v);
  out[i] = hi;
  if (lo) lo[i] = from_f<T>(v - to_f(hi));
}

// Synchronisation of the threads running attn_run: the whole CTA, or the
// four epilogue warps of the per-layer kernel (named barrier 1).
struct SyncCta {
  __device__ __forceinline__ void operator()() const { __syncthreads(); }
};
struct SyncEpilogueWarps {
  __device__ __forceinline__ void operator()() const { asm volatile("bar.sync 1, 128;" ::: "memory"); }
};

template <typename T>
struct AttnArgs {
  const float* q;
  const int32_t* rows;
  const int32_t* count;
  int n, nq, nkv;
  const int32_t* len;
  const int64_t* seq_off;
  const int32_t* cap;
  const T* Kc;
  const T* Vc;
  int max_spans;
  float* part_m;
  float* part_l;
  float* part_acc;
  int32_t* ctr;
  T* out;
  T* out_lo;
  const int32_t* status;
};

// Dynamic shared memory used by attn_run (bytes): double-buffered K (rows
// padded by 16 bytes) and V chunks, the scaled queries, the logits, the
// probabilities by position, the row prefix and the rows' cache offsets,
// positions and head strides.
template <typename T, int HD>
__host__ __device__ constexpr size_t attn_smem_fixed() {
  return 2 * (size_t)kChunk * (HD + 16 / sizeof(T)) * sizeof(T) + 2 * (size_t)kChunk * HD * sizeof(T);
}
inline size_t attn_smem_bytes(size_t fixed, int G, int hd, int max_spans, int max_rows) {
  const int gp = G <= 1 ? 1 : (G <= 2 ? 2 : (G <= 4 ? 4 : 8));
  (void)max_spans;
  return fixed + (size_t)gp * hd * 4 + 2 * (size_t)gp * kChunk * 4 + (size_t)(max_rows + 1) * 4 + 8 +
         (size_t)max_rows * 16;
}

// Merge of a (row j, KV head g)'s nsp span partials, by the CTA that
// completed it (NT threads numbered tid), in span order: the tpo adjacent
// threads of an output (four consecutive channels of one head) take spans
// sub, sub + tpo, ... with a running rescaled sum (running max M, sum L, output
// a), loading D of their spans' partials at a time; the tpo results are then
// combined by a lane butterfly (every thread ends with the same values).  When
// the outputs outnumber the threads, the threads take them in rounds of NT.
// B2: the partial maxima are base-2 logarithms (weights 2^(m - M)).
template <typename T, int HD, int NT, bool B2 = false>
__device__ __forceinline__ void attn_span_merge(const AttnArgs<T>& A, int j, int g, int nsp, size_t obase, int tid) {
  auto ex = [](float x) { return B2 ? exp2f(x) : expf(x); };
  constexpr int D = NT >= 256 ? 16 : 8;   // partials in flight per thread
  const int nq = A.nq, G = A.nq / A.nkv, max_spans = A.max_spans;
  const float* __restrict__ part_acc = A.part_acc;
  const float* __restrict__ part_m = A.part_m;
  const float* __restrict__ part_l = A.part_l;
  T* __restrict__ out = A.out;
  T* __restrict__ out_lo = A.out_lo;
  const int n4 = G * HD / 4;
  int tpo = 1;
  while (tpo < 8 && tpo * 2 * n4 <= NT) tpo *= 2;
  const int nwork = (n4 * tpo + 31) & ~31;   // whole warps take part in the butterfly
  constexpr int kRounds = (8 * HD / 4 + NT - 1) / NT;   // at most 8 query heads per KV head
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int w = tid + r * NT;
    if (w >= nwork) break;
    const int x4 = w / tpo, sub = w % tpo;
    const bool act = x4 < n4;
    const int h = act ? (x4 * 4) / HD : 0, ee = act ? x4 * 4 - h * HD : 0;
    const size_t hb = ((size_t)j * nq + g * G + h) * max_spans;
    float M = -INFINITY, L = 0.f;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c0 = sub; act && c0 < nsp; c0 += D * tpo) {
      float4 t[D];
      float ms[D], ls[D];
#pragma unroll
      for (int k = 0; k < D; ++k) {
        const int cc = c0 + k * tpo;
        if (cc < nsp) {
          t[k] = __ldcg(reinterpret_cast<const float4*>(part_acc + (hb + cc) * HD + ee));
          ms[k] = __ldcg(part_m + hb + cc);
          ls[k] = __ldcg(part_l + hb + cc);
        }
      }
#pragma unroll
      for (int k = 0; k < D; ++k) {
        if (c0 + k * tpo < nsp) {
          const float mn = fmaxf(M, ms[k]);
          const float fo = ex(M - mn), fn = ex(ms[k] - mn);
          a.x = a.x * fo + t[k].x * fn;
          a.y = a.y * fo + t[k].y * fn;
          a.z = a.z * fo + t[k].z * fn;
          a.w = a.w * fo + t[k].w * fn;
          L = L * fo + ls[k] * fn;
          M = mn;
        }
      }
    }
    for (int o = 1; o < tpo; o <<= 1) {
      const float M2 = __shfl_xor_sync(0xffffffffu, M, o), L2 = __shfl_xor_sync(0xffffffffu, L, o);
      const float ax = __shfl_xor_sync(0xffffffffu, a.x, o), ay = __shfl_xor_sync(0xffffffffu, a.y, o);
      const float az = __shfl_xor_sync(0xffffffffu, a.z, o), aw = __shfl_xor_sync(0xffffffffu, a.w, o);
      const float mn = fmaxf(M, M2);
      const float f1 = M == -INFINITY ? 0.f : ex(M - mn), f2 = M2 == -INFINITY ? 0.f : ex(M2 - mn);
      a.x = a.x * f1 + ax * f2;
      a.y = a.y * f1 + ay * f2;
      a.z = a.z * f1 + az * f2;
      a.w = a.w * f1 + aw * f2;
      L = L * f1 + L2 * f2;
      M = mn;
    }
    if (act && sub == 0) {
      const size_t o = obase + (size_t)h * HD + ee;
      store_out(out, out_lo, o + 0, a.x / L);
      store_out(out, out_lo, o + 1, a.y / L);
      store_out(out, out_lo, o + 2, a.z / L);
      store_out(out, out_lo, o + 3, a.w / L);
    }
  }
}

// Query heads per KV head rounded up to 1, 2, 4 or 8 (the work-loop template).
inline int attn_group_pad(int G) { return G <= 1 ? 1 : (G <= 2 ? 2 : (G <= 4 ? 4 : 8)); }

// Processes this CTA's share (items cta, cta + ncta, ...) of one layer's
// attention with NT threads numbered tid; `sync` synchronises them;
// `sc` points to 32 floats of shared scratch.  With `pdl` the copies that do
// not depend on the preceding kernel start before waiting on it.  GP >= G is
// the padded number of query heads per KV head.
//
// Thread mapping within a 64-position chunk:
//   logits: a warp scores 16 positions (32 for one head), 32 / GP positions x GP
//           heads per round: lane l multiplies dims HD/32 * l.. of each K row with
//           the same dims of the queries (held in registers), and a halving
//           butterfly over the lanes leaves the full dot product of
//           (position l / GP, head l % GP) in lane l;
//   P.V:    thread t owns channels 8 * (t % (HD/8)) .. +8 of every head for the
//           positions of group t / (HD/8); its partial sums stay in registers
//           across the chunks of the span (rescaled by the online-softmax
//           factor) and the groups are summed once at the end of the span.
template <typename T, int HD, int GP, int NT, typename Sync>
__device__ __forceinline__ void attn_run(const AttnArgs<T>& A, int tid, int cta, int ncta, uint8_t* smem,
                                         float* sc, Sync sync, bool pdl) {
  static_assert(GP == 1 || GP == 2 || GP == 4 || GP == 8, "GP");
  static_assert(HD == 64 || HD == 128, "HD");
  const float* __restrict__ q = A.q;
  const int32_t* rows = A.rows;
  const int32_t* count = A.count;
  const int n = A.n, nq = A.nq, nkv = A.nkv;
  const int32_t* len = A.len;
  const int64_t* seq_off = A.seq_off;
  const int32_t* cap = A.cap;
  const T* __restrict__ Kc = A.Kc;
  const T* __restrict__ Vc = A.Vc;
  const int max_spans = A.max_spans;
  float* __restrict__ part_m = A.part_m;
  float* __restrict__ part_l = A.part_l;
  float* __restrict__ part_acc = A.part_acc;
  int32_t* ctr = A.ctr;
  T* __restrict__ out = A.out;
  T* __restrict__ out_lo = A.out_lo;
  const int32_t* status = A.status;
  // Rows, counts and positions were written by kernels that completed before
  // the preceding kernel started, and cache positions below len[i] by earlier
  // steps: the work decomposition and the first chunk's copies can start
  // before waiting on the preceding kernel (which writes q and the new
  // token's K/V at position len[i]).
  const int aborted = *reinterpret_cast<const volatile int32_t*>(status + 1);
  const int m = count ? *count : n;
  if (aborted != 0 || m <= 0) {
    if (pdl) pdl_wait();
    return;
  }
  constexpr int PAD = 16 / sizeof(T);           // one 16-byte slot of padding per K row
  constexpr int KROW = HD + PAD;
  constexpr int V16 = HD * (int)sizeof(T) / 16;  // 16-byte pieces per row
  constexpr int E16 = 16 / sizeof(T);            // elements per piece
  constexpr int CH = HD / 8;                     // P.V channel groups of 8
  constexpr int NPG = NT / CH;                   // P.V position groups
  constexpr int NW = NT / 32;                    // warps
  constexpr int PPG = kChunk / NPG;              // positions per group and chunk
  const int G = nq / nkv;
  T* Kb0 = reinterpret_cast<T*>(smem);                          // 2 x [kChunk][KROW]
  T* Vb0 = Kb0 + 2 * kChunk * KROW;                             // 2 x [kChunk][HD]
  float* qs = reinterpret_cast<float*>(Vb0 + 2 * kChunk * HD);  // [GP][HD]
  float* lg = qs + GP * HD;                                     // [GP][kChunk] logits
  float* pt = lg + GP * kChunk;                                 // [kChunk][GP] probabilities
  int* pref = reinterpret_cast<int*>(pt + GP * kChunk);         // [m + 1] span prefix over rows
  int64_t* rbase = reinterpret_cast<int64_t*>(                  // [m] cache offset of each row
      (reinterpret_cast<uintptr_t>(pref + m + 1) + 7) & ~uintptr_t(7));
  int* rnp = reinterpret_cast<int*>(rbase + m);                 // [m] positions (len + 1)
  int* rhs = rnp + m;                                           // [m] head stride (cap * HD)
  float* red = reinterpret_cast<float*>(Kb0);                   // [NPG][HR][HD], after the last chunk
  float* alpha_s = sc;        // [8]
  float* mrun_s = sc + 8;     // [8]
  float* lrun_s = sc + 16;    // [8]
  int* last_s_p = reinterpret_cast<int*>(sc + 24);
  int* span_s_p = reinterpret_cast<int*>(sc + 25);

  const int warp = tid >> 5, lane = tid & 31;
  // positions per row (kept in pref[1..m]) and their total -> span length P
  if (warp == 0) {
    long long tot = 0;
    for (int j = lane; j < m; j += 32) {
      const int i = rows ? rows[j] : j;
      const int np = len[i] + 1;
      rnp[j] = np;
      rbase[j] = seq_off[i] * nkv * HD;
      rhs[j] = cap[i] * HD;
      pref[j + 1] = np;
      tot += np;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    __syncwarp();
    // about one item per CTA, at least one chunk per span
    const long long want = (tot * nkv + ncta - 1) / ncta;
    const int P0 = (int)min((long long)kMaxSpan, max((long long)kChunk, want));
    const int P = (P0 + kChunk - 1) / kChunk * kChunk;
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
  sync();
  const int P = *span_s_p;
  const int total = pref[m] * nkv;
  const float scale = rsqrtf((float)HD);
  bool waited = !pdl;
  const int cg = tid % CH, pg = tid / CH;                 // P.V: channel group, position group

  for (int item = cta; item < total; item += ncta) {
    const int g = item % nkv;
    const int js = item / nkv;
    int lo = 0, hi = m;   // j with pref[j] <= js < pref[j+1]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pref[mid] <= js) lo = mid;
      else hi = mid;
    }
    const int j = lo, sp = js - pref[j];
    const int npos = rnp[j];
    const int nsp = pref[j + 1] - pref[j];
    const int s0 = sp * P, s1 = min(npos, s0 + P);
    const int nch = (s1 - s0 + kChunk - 1) / kChunk;
    const int64_t kvo = rbase[j] + (int64_t)g * rhs[j];   // kv_offset of (row j's sequence, head g, position 0)
    const T* Kbase = Kc + kvo;
    const T* Vbase = Vc + kvo;

    auto issue = [&](int c) {   // chunk c of this span into buffer c & 1
      const int p0 = s0 + c * kChunk, cnt = min(kChunk, s1 - p0);
      T* Kd = Kb0 + (c & 1) * kChunk * KROW;
      T* Vd = Vb0 + (c & 1) * kChunk * HD;
      for (int x = tid; x < cnt * V16; x += NT) {
        const int p = x / V16, s = x - p * V16;
        cp_async16(Kd + p * KROW + s * E16, Kbase + (size_t)(p0 + p) * HD + s * E16);
        cp_async16(Vd + p * HD + s * E16, Vbase + (size_t)(p0 + p) * HD + s * E16);
      }
      cp_async_commit();
    };
    if (!waited) {
      // the first chunk may be copied before the wait unless it holds the new
      // token (position len[i] = npos - 1)
      const bool has_new = s0 + min(kChunk, s1 - s0) >= npos;
      if (!has_new) issue(0);
      pdl_wait();
      pdl_trigger();
      waited = true;
      if (has_new) issue(0);
    } else {
      issue(0);
    }
    const float* qj = q + (size_t)j * nq * HD + (size_t)g * G * HD;
    for (int x = tid; x < GP * HD; x += NT) qs[x] = x < G * HD ? qj[x] * scale : 0.f;
    sync();
    // this lane's query dims for the logits
    constexpr int DPL = HD / 32;
    float qr[GP][DPL];
#pragma unroll
    for (int h = 0; h < GP; ++h)
#pragma unroll
      for (int d = 0; d < DPL; ++d) qr[h][d] = qs[h * HD + lane * DPL + d];
    if (tid < GP) {
      mrun_s[tid] = -INFINITY;
      lrun_s[tid] = 0.f;
    }
    float acc[GP][8];
#pragma unroll
    for (int h = 0; h < GP; ++h)
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[h][k] = 0.f;

    for (int c = 0; c < nch; ++c) {
      if (c + 1 < nch) {
        issue(c + 1);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      sync();
      const int cnt = min(kChunk, s1 - (s0 + c * kChunk));
      const T* Ks = Kb0 + (c & 1) * kChunk * KROW;
      const T* Vs = Vb0 + (c & 1) * kChunk * HD;
      // logits: rounds of PPR positions x GP heads per warp, reduced over the lanes
      {
        constexpr int PPR = 32 / GP;                                    // positions per round
        constexpr int PPW = kChunk / NW > PPR ? kChunk / NW : PPR;      // positions per warp
        constexpr int ROUNDS = PPW / PPR;
        const int pw = warp * PPW;
        if (pw < kChunk) {
#pragma unroll
          for (int r = 0; r < ROUNDS; ++r) {
            const int pb = pw + r * PPR;
            float v[32];
#pragma unroll
            for (int pi = 0; pi < PPR; ++pi) {
              const int p = pb + pi;
              float kd[DPL];
              if (p < cnt) {
                if (DPL == 4) {
                  const uint2 u = *reinterpret_cast<const uint2*>(Ks + p * KROW + lane * 4);
                  if (sizeof(T) == 2) {
                    kd[0] = __uint_as_float(u.x << 16); kd[1] = __uint_as_float(u.x & 0xFFFF0000u);
                    kd[2] = __uint_as_float(u.y << 16); kd[3] = __uint_as_float(u.y & 0xFFFF0000u);
                  }
                }
                if (sizeof(T) == 4 || DPL != 4) {
#pragma unroll
                  for (int d = 0; d < DPL; ++d) kd[d] = to_f(Ks[p * KROW + lane * DPL + d]);
                }
              } else {
#pragma unroll
                for (int d = 0; d < DPL; ++d) kd[d] = 0.f;
              }
#pragma unroll
              for (int h = 0; h < GP; ++h) {
                float a = 0.f;
#pragma unroll
                for (int d = 0; d < DPL; ++d) a += qr[h][d] * kd[d];
                v[pi * GP + h] = a;
              }
            }
            // halving butterfly: lane l ends with the sum of value l
#pragma unroll
            for (int o = 16, nv = 16; o >= 1; o >>= 1, nv >>= 1) {
              const bool upper = (lane & o) != 0;
#pragma unroll
              for (int x = 0; x < nv; ++x) {
                const float send = upper ? v[x] : v[x + nv];
                const float keep = upper ? v[x + nv] : v[x];
                v[x] = keep + __shfl_xor_sync(0xffffffffu, send, o);
              }
            }
            const int p = pb + lane / GP, h = lane % GP;
            lg[h * kChunk + p] = p < cnt ? v[0] : -INFINITY;
          }
        }
      }
      sync();
      // online softmax update, one warp per head; probabilities stored by position
      for (int h = warp; h < G; h += NW) {
        const float v0 = lg[h * kChunk + lane], v1 = lg[h * kChunk + lane + 32];
        const float mc = warp_max(fmaxf(v0, v1));
        const float mo = mrun_s[h];
        const float mn = fmaxf(mo, mc);
        const float e0 = (lane < cnt) ? expf(v0 - mn) : 0.f;
        const float e1 = (lane + 32 < cnt) ? expf(v1 - mn) : 0.f;
        pt[lane * GP + h] = e0;
        pt[(lane + 32) * GP + h] = e1;
        const float sv = warp_sum(e0 + e1);
        if (lane == 0) {
          const float al = (mo == -INFINITY) ? 0.f : expf(mo - mn);
          alpha_s[h] = al;
          mrun_s[h] = mn;
          lrun_s[h] = lrun_s[h] * al + sv;
        }
      }
      for (int x = tid; x < (GP - G) * kChunk; x += NT) {   // padded heads
        const int h = G + x / kChunk, p = x % kChunk;
        pt[p * GP + h] = 0.f;
        if (p == 0) alpha_s[h] = 0.f;
      }
      sync();
      // P.V: channels 8*cg.. of every head over the positions of group pg
      {
        float al[GP];
#pragma unroll
        for (int h = 0; h < GP; ++h) al[h] = alpha_s[h];
#pragma unroll
        for (int h = 0; h < GP; ++h)
#pragma unroll
          for (int k = 0; k < 8; ++k) acc[h][k] *= al[h];
#pragma unroll
        for (int u = 0; u < PPG; ++u) {
          const int p = pg * PPG + u;
          if (p < cnt) {
            float v8[8];
            load8s<T>(Vs + p * HD + cg * 8, v8);
            float pv[GP];
            if (GP >= 4) {
#pragma unroll
              for (int h4 = 0; h4 < GP; h4 += 4) {
                const float4 t4 = *reinterpret_cast<const float4*>(pt + p * GP + h4);
                pv[h4] = t4.x; pv[h4 + 1] = t4.y; pv[h4 + 2] = t4.z; pv[h4 + 3] = t4.w;
              }
            } else {
#pragma unroll
              for (int h = 0; h < GP; ++h) pv[h] = pt[p * GP + h];
            }
#pragma unroll
            for (int h = 0; h < GP; ++h)
#pragma unroll
              for (int k = 0; k < 8; ++k) acc[h][k] += pv[h] * v8[k];
          }
        }
      }
      sync();   // buffer (c & 1) is refilled by the issue of chunk c + 2
    }
    // sum the position groups (the K and V buffers are free now), in passes
    // of HR heads when [NPG][GP][HD] floats do not fit there
    constexpr size_t kKVBytes = 2 * (size_t)kChunk * KROW * sizeof(T) + 2 * (size_t)kChunk * HD * sizeof(T);
    constexpr int HR = (size_t)NPG * GP * HD * 4 <= kKVBytes
                           ? GP
                           : ((size_t)NPG * (GP / 2) * HD * 4 <= kKVBytes ? GP / 2 : (GP >= 4 ? GP / 4 : 1));
    static_assert((size_t)NPG * HR * HD * 4 <= kKVBytes, "attention reduction buffer");
    const size_t obase = (size_t)j * nq * HD + (size_t)g * G * HD;
#pragma unroll
    for (int h0 = 0; h0 < GP; h0 += HR) {
      if (h0 > 0) sync();   // the previous pass has read the buffer
#pragma unroll
      for (int hh = 0; hh < HR; ++hh) {
        float4* r = reinterpret_cast<float4*>(red + ((size_t)pg * HR + hh) * HD + cg * 8);
        r[0] = make_float4(acc[h0 + hh][0], acc[h0 + hh][1], acc[h0 + hh][2], acc[h0 + hh][3]);
        r[1] = make_float4(acc[h0 + hh][4], acc[h0 + hh][5], acc[h0 + hh][6], acc[h0 + hh][7]);
      }
      sync();
      for (int x = tid; x < HR * HD; x += NT) {
        const int hh = x / HD, e = x - hh * HD, h = h0 + hh;
        if (h >= G) continue;
        float o = 0.f;
#pragma unroll
        for (int q2 = 0; q2 < NPG; ++q2) o += red[((size_t)q2 * HR + hh) * HD + e];
        if (nsp == 1) {
          store_out(out, out_lo, obase + (size_t)h * HD + e, o / lrun_s[h]);
        } else {
          const size_t slot = ((size_t)j * nq + g * G + h) * max_spans + sp;
          __stcg(part_acc + slot * HD + e, o);
          if (e == 0) {
            __stcg(part_m + slot, mrun_s[h]);
            __stcg(part_l + slot, lrun_s[h]);
          }
        }
      }
    }
    if (nsp > 1) {
      sync();
      if (tid == 0) {
        __threadfence();
        const int old = atomicAdd(&ctr[j * nkv + g], 1);
        *last_s_p = (old == nsp - 1);
        if (*last_s_p) ctr[j * nkv + g] = 0;
        __threadfence();
      }
      sync();
      if (*last_s_p) attn_span_merge<T, HD, NT>(A, j, g, nsp, obase, tid);
    }
    sync();
  }
  if (!waited) {
    pdl_wait();
    pdl_trigger();
  }
}

}  // namespace buddy

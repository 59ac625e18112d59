// Decode attention work loop shared by the attention kernel and the
// per-layer persistent kernel (see attention.cu for the algorithm).
#pragma once

#include <cuda_runtime.h>

#include <algorithm>

#include "common.cuh"

namespace buddy {

constexpr int kChunk = 64;
constexpr int kAttnThreads = 128;
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

// Dynamic shared memory used by attn_run (bytes).
template <typename T, int HD>
__host__ __device__ constexpr size_t attn_smem_fixed() {
  return 2 * (size_t)kChunk * (HD + 16 / sizeof(T)) * sizeof(T) + 2 * (size_t)kChunk * HD * sizeof(T);
}
inline size_t attn_smem_bytes(size_t fixed, int G, int hd, int max_spans, int max_rows) {
  return fixed + (size_t)G * hd * 4 + (size_t)G * kChunk * 4 + (size_t)G * hd * 4 + (size_t)G * max_spans * 4 +
         (size_t)(max_rows + 1) * 4;
}

// Processes this CTA's share (items cta, cta + ncta, ...) of one layer's
// attention with kAttnThreads threads numbered tid; `sync` synchronises them;
// `sc` points to 32 floats of shared scratch.  With `pdl` the copies that do
// not depend on the preceding kernel start before waiting on it.
template <typename T, int HD, typename Sync>
__device__ __forceinline__ void attn_run(const AttnArgs<T>& A, int tid, int cta, int ncta, uint8_t* smem,
                                         float* sc, Sync sync, bool pdl) {
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
  if (*reinterpret_cast<const volatile int32_t*>(status + 1) != 0) {
    if (pdl) pdl_wait();
    return;
  }
  const int m = count ? *count : n;
  if (m <= 0) {
    if (pdl) pdl_wait();
    return;
  }
  constexpr int PAD = 16 / sizeof(T);           // one 16-byte slot of padding per K row
  constexpr int KROW = HD + PAD;
  constexpr int V16 = HD * (int)sizeof(T) / 16;  // 16-byte pieces per row
  constexpr int E16 = 16 / sizeof(T);            // elements per piece
  const int G = nq / nkv;
  T* Kb0 = reinterpret_cast<T*>(smem);                          // 2 x [kChunk][KROW]
  T* Vb0 = Kb0 + 2 * kChunk * KROW;                              // 2 x [kChunk][HD]
  float* qs = reinterpret_cast<float*>(Vb0 + 2 * kChunk * HD);   // [G][HD]
  float* ps = qs + G * HD;                                       // [G][kChunk]
  float* red = ps + G * kChunk;                                  // [G][HD] second-half sums (HD = 64)
  float* wch = red + G * HD;                                     // [G][max_spans] merge weights
  int* pref = reinterpret_cast<int*>(wch + G * max_spans);       // [m + 1] span prefix over rows
  float* alpha_s = sc;        // [8]
  float* mrun_s = sc + 8;     // [8]
  float* lrun_s = sc + 16;    // [8]
  int* last_s_p = reinterpret_cast<int*>(sc + 24);
  int* span_s_p = reinterpret_cast<int*>(sc + 25);

  const int warp = tid >> 5, lane = tid & 31;
  // total positions -> span length P (the same value in every CTA)
  if (warp == 0) {
    long long tot = 0;
    for (int j = lane; j < m; j += 32) tot += len[rows ? rows[j] : j] + 1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    if (lane == 0) {
      const long long items = max(1, ncta / 2);
      const long long want = (tot * nkv + items - 1) / items;
      const int P = (int)min((long long)kMaxSpan, max((long long)kChunk, want));
      *span_s_p = (P + kChunk - 1) / kChunk * kChunk;
    }
  }
  sync();
  const int P = *span_s_p;
  if (warp == 0) {
    int carry = 0;
    for (int b = 0; b < m; b += 32) {
      const int j = b + lane;
      int ns = 0;
      if (j < m) ns = (len[rows ? rows[j] : j] + 1 + P - 1) / P;
      int x = ns;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (j < m) pref[j + 1] = carry + x;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) pref[0] = 0;
  }
  sync();
  const int total = pref[m] * nkv;
  const float scale = rsqrtf((float)HD);
  bool waited = !pdl;
  constexpr int SPLIT = kAttnThreads / HD;   // 1 for HD = 128, 2 for HD = 64
  const int e = tid % HD, half = tid / HD;

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
    const int i = rows ? rows[j] : j;
    const int npos = len[i] + 1;
    const int nsp = pref[j + 1] - pref[j];
    const int s0 = sp * P, s1 = min(npos, s0 + P);
    const int nch = (s1 - s0 + kChunk - 1) / kChunk;
    const T* Kbase = Kc + kv_offset(seq_off, cap, i, nkv, HD, g, 0);
    const T* Vbase = Vc + kv_offset(seq_off, cap, i, nkv, HD, g, 0);

    auto issue = [&](int c) {   // chunk c of this span into buffer c & 1
      const int p0 = s0 + c * kChunk, cnt = min(kChunk, s1 - p0);
      T* Kd = Kb0 + (c & 1) * kChunk * KROW;
      T* Vd = Vb0 + (c & 1) * kChunk * HD;
      for (int x = tid; x < cnt * V16; x += kAttnThreads) {
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
    for (int x = tid; x < G * HD; x += kAttnThreads) qs[x] = qj[x] * scale;
    if (tid < G) {
      mrun_s[tid] = -INFINITY;
      lrun_s[tid] = 0.f;
    }
    float acc[8];
#pragma unroll
    for (int h = 0; h < 8; ++h) acc[h] = 0.f;

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
      // logits: 32 consecutive pairs of a warp share the head, differ in position
      for (int x = tid; x < G * kChunk; x += kAttnThreads) {
        const int h = x / kChunk, p = x - h * kChunk;
        float a = -INFINITY;
        if (p < cnt) {
          a = 0.f;
          const T* kr = Ks + p * KROW;
          const float* qh = qs + h * HD;
#pragma unroll 4
          for (int ee = 0; ee < HD; ee += 8) {
            float kv[8];
            load8s<T>(kr + ee, kv);
            const float4 q0 = *reinterpret_cast<const float4*>(qh + ee);
            const float4 q1 = *reinterpret_cast<const float4*>(qh + ee + 4);
            a += kv[0] * q0.x + kv[1] * q0.y + kv[2] * q0.z + kv[3] * q0.w + kv[4] * q1.x + kv[5] * q1.y +
                 kv[6] * q1.z + kv[7] * q1.w;
          }
        }
        ps[x] = a;
      }
      sync();
      // online softmax update, one warp per head
      for (int h = warp; h < G; h += kAttnThreads / 32) {
        const float v0 = ps[h * kChunk + lane], v1 = ps[h * kChunk + lane + 32];
        const float mc = warp_max(fmaxf(v0, v1));
        const float mo = mrun_s[h];
        const float mn = fmaxf(mo, mc);
        const float e0 = (lane < cnt) ? expf(v0 - mn) : 0.f;
        const float e1 = (lane + 32 < cnt) ? expf(v1 - mn) : 0.f;
        ps[h * kChunk + lane] = e0;
        ps[h * kChunk + lane + 32] = e1;
        const float sv = warp_sum(e0 + e1);
        if (lane == 0) {
          const float al = (mo == -INFINITY) ? 0.f : expf(mo - mn);
          alpha_s[h] = al;
          mrun_s[h] = mn;
          lrun_s[h] = lrun_s[h] * al + sv;
        }
      }
      sync();
      // P.V with rescaling of the running output
      const int pa = half * (kChunk / SPLIT), pb = min(cnt, pa + kChunk / SPLIT);
#pragma unroll
      for (int h = 0; h < 8; ++h)
        if (h < G) acc[h] *= alpha_s[h];
      for (int p = pa; p < pb; ++p) {
        const float v = to_f(Vs[p * HD + e]);
#pragma unroll
        for (int h = 0; h < 8; ++h)
          if (h < G) acc[h] += ps[h * kChunk + p] * v;
      }
      sync();   // buffer (c & 1) is refilled by the issue of chunk c + 2
    }
    if (SPLIT == 2) {
      if (half == 1)
        for (int h = 0; h < G; ++h) red[h * HD + e] = acc[h];
      sync();
      if (half == 0)
        for (int h = 0; h < G; ++h) acc[h] += red[h * HD + e];
    }
    const size_t obase = (size_t)j * nq * HD + (size_t)g * G * HD;
    if (nsp == 1) {
      if (half == 0)
        for (int h = 0; h < G; ++h) store_out(out, out_lo, obase + (size_t)h * HD + e, acc[h] / lrun_s[h]);
    } else {
      if (half == 0) {
        for (int h = 0; h < G; ++h) {
          const size_t slot = ((size_t)j * nq + g * G + h) * max_spans + sp;
          __stcg(part_acc + slot * HD + e, acc[h]);
          if (e == 0) {
            __stcg(part_m + slot, mrun_s[h]);
            __stcg(part_l + slot, lrun_s[h]);
          }
        }
      }
      sync();
      if (tid == 0) {
        __threadfence();
        const int old = atomicAdd(&ctr[j * nkv + g], 1);
        *last_s_p = (old == nsp - 1);
        if (*last_s_p) ctr[j * nkv + g] = 0;
        __threadfence();
      }
      sync();
      if (*last_s_p) {
        // merge in span order: per head the weights exp(m_s - M), then every
        // output channel as independent loads over the spans
        for (int h = warp; h < G; h += kAttnThreads / 32) {
          const size_t base = ((size_t)j * nq + g * G + h) * max_spans;
          float mloc = -INFINITY;
          for (int cc = lane; cc < nsp; cc += 32) mloc = fmaxf(mloc, __ldcg(part_m + base + cc));
          const float M = warp_max(mloc);
          float lsum = 0.f;
          for (int cc = lane; cc < nsp; cc += 32) {
            const float w = expf(__ldcg(part_m + base + cc) - M);
            wch[h * max_spans + cc] = w;
            lsum += __ldcg(part_l + base + cc) * w;
          }
          lsum = warp_sum(lsum);
          if (lane == 0) lrun_s[h] = lsum;
        }
        sync();
        // four consecutive channels per thread; the partials of eight spans
        // are loaded together, then accumulated in span order
        for (int x4 = tid; x4 < G * HD / 4; x4 += kAttnThreads) {
          const int h = (x4 * 4) / HD, ee = x4 * 4 - h * HD;
          const float* pa0 = part_acc + ((size_t)j * nq + g * G + h) * max_spans * HD + ee;
          const float* wh = wch + h * max_spans;
          float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
          for (int c0 = 0; c0 < nsp; c0 += 8) {
            float4 t[8];
#pragma unroll
            for (int k = 0; k < 8; ++k)
              if (c0 + k < nsp) t[k] = __ldcg(reinterpret_cast<const float4*>(pa0 + (size_t)(c0 + k) * HD));
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              if (c0 + k < nsp) {
                const float w = wh[c0 + k];
                a.x += t[k].x * w;
                a.y += t[k].y * w;
                a.z += t[k].z * w;
                a.w += t[k].w * w;
              }
            }
          }
          const float l = lrun_s[h];
          const size_t o = obase + (size_t)h * HD + ee;
          store_out(out, out_lo, o + 0, a.x / l);
          store_out(out, out_lo, o + 1, a.y / l);
          store_out(out, out_lo, o + 2, a.z / l);
          store_out(out, out_lo, o + 3, a.w / l);
        }
      }
    }
    sync();
  }
  if (!waited) {
    pdl_wait();
    pdl_trigger();
  }
}

}  // namespace buddy

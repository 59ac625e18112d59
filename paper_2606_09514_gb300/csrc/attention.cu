// Decode attention for one layer (Eq. 9): for every active row j (sequence
// i = rows[j]) and KV head g, the G = n_q / n_kv query heads of the group
// attend over positions 0..len[i] of that head's cache (the new token included;
// zero-filled positions of earlier skipped steps take part with logit 0).
//
// Work items are (row, chunk of kChunk positions, KV head), enumerated on the
// device from the rows' lengths; persistent CTAs walk them.  A CTA stages the
// chunk's K and V in shared memory with 16-byte cp.async copies (K rows padded
// so that lanes reading 32 different positions hit distinct banks), computes
// the G x chunk logits, a chunk-local softmax and P.V in fp32, and writes a
// partial (running max, sum of exponentials, unnormalised output).  The last
// CTA to finish a (row, head) merges its chunks in chunk order (log-sum-exp)
// and writes the attention output in the GEMM input type.
#include <cuda_runtime.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace buddy {

constexpr int kChunk = 64;
constexpr int kAttnThreads = 128;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
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

template <typename T, int HD>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(
    const float* __restrict__ q, const int32_t* rows, const int32_t* count, int n, int nq, int nkv,
    const int32_t* len, const int64_t* seq_off, const int32_t* cap, const T* __restrict__ Kc,
    const T* __restrict__ Vc, int max_chunks, float* __restrict__ part_m, float* __restrict__ part_l,
    float* __restrict__ part_acc, int32_t* ctr, T* __restrict__ out, T* __restrict__ out_lo,
    const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int m = count ? *count : n;
  if (m <= 0) return;
  constexpr int PAD = 16 / sizeof(T);          // one 16-byte slot of padding per K row
  constexpr int KROW = HD + PAD;
  constexpr int V16 = HD * (int)sizeof(T) / 16; // 16-byte pieces per row
  const int G = nq / nkv;
  extern __shared__ __align__(16) uint8_t smraw[];
  T* Ks = reinterpret_cast<T*>(smraw);                           // [kChunk][KROW]
  T* Vs = Ks + kChunk * KROW;                                     // [kChunk][HD]
  float* qs = reinterpret_cast<float*>(Vs + kChunk * HD);         // [G][HD]
  float* ps = qs + G * HD;                                        // [G][kChunk]
  float* wch = ps + G * kChunk;                                   // [G][max_chunks] merge weights
  int* pref = reinterpret_cast<int*>(wch + G * max_chunks);       // [m + 1] chunk prefix over rows
  __shared__ float mx_s[8], sum_s[8];
  __shared__ int last_s;

  // chunk counts and their prefix over the active rows
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (warp == 0) {
    int carry = 0;
    for (int b = 0; b < m; b += 32) {
      const int j = b + lane;
      int nc = 0;
      if (j < m) nc = (len[rows ? rows[j] : j] + 1 + kChunk - 1) / kChunk;
      int x = nc;
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
  __syncthreads();
  const int total = pref[m] * nkv;
  const float scale = rsqrtf((float)HD);

  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    const int g = item % nkv;
    const int jc = item / nkv;
    int lo = 0, hi = m;   // find j with pref[j] <= jc < pref[j+1]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pref[mid] <= jc) lo = mid;
      else hi = mid;
    }
    const int j = lo, c = jc - pref[j];
    const int i = rows ? rows[j] : j;
    const int npos = len[i] + 1;
    const int nch = pref[j + 1] - pref[j];
    const int p0 = c * kChunk, cnt = min(kChunk, npos - p0);
    const T* Kb = Kc + kv_offset(seq_off, cap, i, nkv, HD, g, p0);
    const T* Vb = Vc + kv_offset(seq_off, cap, i, nkv, HD, g, p0);
    for (int x = tid; x < cnt * V16; x += kAttnThreads) {
      const int p = x / V16, s = x - p * V16;
      cp_async16(Ks + p * KROW + s * (16 / sizeof(T)), Kb + (size_t)p * HD + s * (16 / sizeof(T)));
      cp_async16(Vs + p * HD + s * (16 / sizeof(T)), Vb + (size_t)p * HD + s * (16 / sizeof(T)));
    }
    const float* qj = q + (size_t)j * nq * HD + (size_t)g * G * HD;
    for (int x = tid; x < G * HD; x += kAttnThreads) qs[x] = qj[x] * scale;
    cp_async_wait_all();
    __syncthreads();
    // logits: 32 consecutive pairs of a warp share the head, differ in position
    for (int x = tid; x < G * kChunk; x += kAttnThreads) {
      const int h = x / kChunk, p = x - h * kChunk;
      float a = -INFINITY;
      if (p < cnt) {
        a = 0.f;
        const T* kr = Ks + p * KROW;
        const float* qh = qs + h * HD;
#pragma unroll 4
        for (int e = 0; e < HD; e += 8) {
          float kv[8];
          load8s<T>(kr + e, kv);
          const float4 q0 = *reinterpret_cast<const float4*>(qh + e);
          const float4 q1 = *reinterpret_cast<const float4*>(qh + e + 4);
          a += kv[0] * q0.x + kv[1] * q0.y + kv[2] * q0.z + kv[3] * q0.w + kv[4] * q1.x + kv[5] * q1.y +
               kv[6] * q1.z + kv[7] * q1.w;
        }
      }
      ps[x] = a;
    }
    __syncthreads();
    for (int h = warp; h < G; h += kAttnThreads / 32) {
      float mv = fmaxf(ps[h * kChunk + lane], ps[h * kChunk + lane + 32]);
      mv = warp_max(mv);
      const float e0 = (lane < cnt) ? expf(ps[h * kChunk + lane] - mv) : 0.f;
      const float e1 = (lane + 32 < cnt) ? expf(ps[h * kChunk + lane + 32] - mv) : 0.f;
      ps[h * kChunk + lane] = e0;
      ps[h * kChunk + lane + 32] = e1;
      const float sv = warp_sum(e0 + e1);
      if (lane == 0) {
        mx_s[h] = mv;
        sum_s[h] = sv;
      }
    }
    __syncthreads();
    // P.V: thread owns channel e (and for HD = 64 one half of the positions)
    constexpr int SPLIT = kAttnThreads / HD;
    const int e = tid % HD, half = tid / HD;
    const int pa = half * (kChunk / SPLIT), pb = min(cnt, pa + kChunk / SPLIT);
    float acc[8];
#pragma unroll
    for (int h = 0; h < 8; ++h) acc[h] = 0.f;
    for (int p = pa; p < pb; ++p) {
      const float v = to_f(Vs[p * HD + e]);
#pragma unroll
      for (int h = 0; h < 8; ++h)
        if (h < G) acc[h] += ps[h * kChunk + p] * v;
    }
    if (SPLIT == 2) {
      __syncthreads();   // ps no longer needed: reuse it for the second half's sums
      float* red = reinterpret_cast<float*>(Ks);
      if (half == 1)
        for (int h = 0; h < G; ++h) red[h * HD + e] = acc[h];
      __syncthreads();
      if (half == 0)
        for (int h = 0; h < G; ++h) acc[h] += red[h * HD + e];
    }
    if (nch == 1) {
      if (half == 0)
        for (int h = 0; h < G; ++h)
          store_out(out, out_lo, (size_t)j * nq * HD + (size_t)(g * G + h) * HD + e, acc[h] / sum_s[h]);
    } else {
      if (half == 0) {
        for (int h = 0; h < G; ++h) {
          const size_t slot = ((size_t)j * nq + g * G + h) * max_chunks + c;
          __stcg(part_acc + slot * HD + e, acc[h]);
          if (e == 0) {
            __stcg(part_m + slot, mx_s[h]);
            __stcg(part_l + slot, sum_s[h]);
          }
        }
      }
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&ctr[j * nkv + g], 1);
        last_s = (old == nch - 1);
        if (last_s) ctr[j * nkv + g] = 0;
        __threadfence();
      }
      __syncthreads();
      if (last_s) {
        __threadfence();
        // merge in chunk order: per head the running-max weights, then every
        // output channel as independent loads over the chunks
        for (int h = warp; h < G; h += kAttnThreads / 32) {
          const size_t base = ((size_t)j * nq + g * G + h) * max_chunks;
          float mloc = -INFINITY;
          for (int cc = lane; cc < nch; cc += 32) mloc = fmaxf(mloc, __ldcg(part_m + base + cc));
          const float M = warp_max(mloc);
          float lsum = 0.f;
          for (int cc = lane; cc < nch; cc += 32) {
            const float w = expf(__ldcg(part_m + base + cc) - M);
            wch[h * max_chunks + cc] = w;
            lsum += __ldcg(part_l + base + cc) * w;
          }
          lsum = warp_sum(lsum);
          if (lane == 0) sum_s[h] = lsum;
        }
        __syncthreads();
        for (int x = tid; x < G * HD; x += kAttnThreads) {
          const int h = x / HD, ee = x - h * HD;
          const float* pa0 = part_acc + ((size_t)j * nq + g * G + h) * max_chunks * HD + ee;
          const float* wh = wch + h * max_chunks;
          float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
          int cc = 0;
          for (; cc + 4 <= nch; cc += 4) {
            a0 += __ldcg(pa0 + (size_t)(cc + 0) * HD) * wh[cc + 0];
            a1 += __ldcg(pa0 + (size_t)(cc + 1) * HD) * wh[cc + 1];
            a2 += __ldcg(pa0 + (size_t)(cc + 2) * HD) * wh[cc + 2];
            a3 += __ldcg(pa0 + (size_t)(cc + 3) * HD) * wh[cc + 3];
          }
          for (; cc < nch; ++cc) a0 += __ldcg(pa0 + (size_t)cc * HD) * wh[cc];
          store_out(out, out_lo, (size_t)j * nq * HD + (size_t)(g * G + h) * HD + ee,
                    ((a0 + a1) + (a2 + a3)) / sum_s[h]);
        }
      }
    }
    __syncthreads();
  }
}

template <typename T, int HD>
static void attn_impl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q,
                      void* out, void* out_lo, cudaStream_t s) {
  const int G = c.nq / c.nkv;
  const size_t smem = (size_t)kChunk * (HD + 16 / sizeof(T)) * sizeof(T) + (size_t)kChunk * HD * sizeof(T) +
                      (size_t)G * HD * 4 + (size_t)G * kChunk * 4 + (size_t)G * c.attn_max_chunks * 4 +
                      (size_t)(c.maxB + 1) * 4;
  static bool attr_set = false;   // one per instantiation
  if (!attr_set) {
    cudaFuncSetAttribute(attn_kernel<T, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    attr_set = true;
  }
  const int grid = c.num_sms * 4;
  launch_k(attn_kernel<T, HD>, grid, kAttnThreads, smem, s, c.pdl, q, sel.rows, sel.count, sel.n, c.nq,
           c.nkv, (const int32_t*)kv.len, kv.seq_off, kv.cap, (const T*)kv.k_cache[layer],
           (const T*)kv.v_cache[layer], c.attn_max_chunks, c.attn_m, c.attn_l, c.attn_acc, c.attn_ctr, (T*)out,
           (T*)out_lo, (const int32_t*)c.status);
}

int attention_chunk() { return kChunk; }

void launch_attention(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q,
                      void* out, void* out_lo, cudaStream_t s) {
  if (c.dtype == BUDDY_DTYPE_BF16) {
    if (c.hd == 128) attn_impl<bf16, 128>(c, sel, kv, layer, q, out, out_lo, s);
    else attn_impl<bf16, 64>(c, sel, kv, layer, q, out, out_lo, s);
  } else {
    if (c.hd == 128) attn_impl<float, 128>(c, sel, kv, layer, q, out, nullptr, s);
    else attn_impl<float, 64>(c, sel, kv, layer, q, out, nullptr, s);
  }
}

}  // namespace buddy

// Non-GEMM kernels of the budget-routed decode step: argument checks, RMSNorm,
// QKV finalisation (bias, RoPE, cache append, pooled-context update), the router (KV-aware pooling + Decision Module + top-k),
// row compaction with zero K/V for skipped layers, and KV prefill.
#include <cuda_runtime.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace buddy {

// ---------------------------------------------------------------------------
// RoPE table: cos/sin of p * theta^(-2j/hd) evaluated in double, stored fp32.
// ---------------------------------------------------------------------------
__global__ void rope_table_kernel(float* c, float* s, int max_pos, int hd, double theta) {
  const int half = hd / 2;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)max_pos * half) return;
  const int p = (int)(idx / half), j = (int)(idx % half);
  const double a = (double)p * pow(theta, -2.0 * (double)j / (double)hd);
  c[idx] = (float)cos(a);
  s[idx] = (float)sin(a);
}

void launch_rope_table(float* c, float* s, int max_pos, int hd, double theta, cudaStream_t st) {
  const int64_t n = (int64_t)max_pos * (hd / 2);
  rope_table_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(c, s, max_pos, hd, theta);
}

// ---------------------------------------------------------------------------
// Argument checks that need device data.  One CTA decides for the whole call
// and publishes the abort flag that every later kernel of the call reads.
// ---------------------------------------------------------------------------
__global__ void step_check_kernel(int B, const int32_t* k, int Lm, int k_min, const int32_t* len,
                                  const int32_t* cap, int extra, int max_pos, const int32_t* layer_len,
                                  int L, int kv_batch, int32_t* status) {
  pdl_wait();
  pdl_trigger();
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  int b = 0;
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    if (k != nullptr) {
      const int ki = k[i];
      if (ki < k_min || ki > Lm) b |= BUDDY_DEV_BAD_BUDGET;
    }
    const int n = len[i];
    if (n < 0 || n + extra > cap[i] || n + extra > max_pos) b |= BUDDY_DEV_BAD_POSITION;
    if (layer_len != nullptr)
      for (int l = 0; l < L; ++l) {
        const int nl = layer_len[(size_t)l * kv_batch + i];
        if (nl < 0 || nl > n) b |= BUDDY_DEV_BAD_POSITION;
      }
  }
  if (b) atomicOr(&bad, b);
  __syncthreads();
  if (threadIdx.x == 0) {
    status[1] = bad ? 1 : 0;
    if (bad) atomicOr(status, bad);
  }
}

void launch_step_check(const Ctx& c, int B, const int32_t* k, const buddy_kv_state& kv, int extra,
                       int32_t* status, cudaStream_t s) {
  const int k_min = c.have_pred ? 0 : 1;   // 0 = "no budget": the Budget Predictor chooses
  launch_k(step_check_kernel, 1, 256, 0, s, c.pdl, B, k, c.Lm, k_min, (const int32_t*)kv.len, kv.cap, extra,
           c.max_pos, (const int32_t*)kv.layer_len, c.L, kv.batch, status);
}

__global__ void kv_check_kernel(int n_seq, const int32_t* ids, int n_new, int batch,
                                const int32_t* len, const int32_t* cap, int max_pos, int32_t* status) {
  // len: the positions the append starts at (len, or the layer's layer_len)
  pdl_wait();
  pdl_trigger();
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  int b = 0;
  for (int j = threadIdx.x; j < n_seq; j += blockDim.x) {
    const int s = ids[j];
    if (s < 0 || s >= batch) {
      b |= BUDDY_DEV_BAD_SEQ;
      continue;
    }
    const int n = len[s];
    if (n < 0 || n + n_new > cap[s] || n + n_new > max_pos) b |= BUDDY_DEV_BAD_POSITION;
  }
  if (b) atomicOr(&bad, b);
  __syncthreads();
  if (threadIdx.x == 0) {
    status[1] = bad ? 1 : 0;
    if (bad) atomicOr(status, bad);
  }
}

void launch_kv_check(const Ctx& c, int n_seq, const int32_t* ids, int n_new, int batch,
                     const int32_t* len, const int32_t* cap, int32_t* status, cudaStream_t s) {
  launch_k(kv_check_kernel, 1, 256, 0, s, c.pdl, n_seq, ids, n_new, batch, len, cap, c.max_pos, status);
}

// ---------------------------------------------------------------------------
// Block-wide sum for 256-thread blocks.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float block_sum_256(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = (l < (int)(blockDim.x >> 5)) ? red[l] : 0.f;
  t = warp_sum(t);
  __syncthreads();
  return t;
}

// ---------------------------------------------------------------------------
// RMSNorm with row gather: xn[j] = act(H[rows[j]] * rsqrt(mean(H^2) + eps) * g)
// ---------------------------------------------------------------------------
// Four consecutive values of a row as one vector store.
__device__ __forceinline__ void store4(float* p, const float* y) {
  *reinterpret_cast<float4*>(p) = make_float4(y[0], y[1], y[2], y[3]);
}
__device__ __forceinline__ void store4(bf16* p, const float* y) {
  const bf16 a = from_f<bf16>(y[0]), b = from_f<bf16>(y[1]), c = from_f<bf16>(y[2]), e = from_f<bf16>(y[3]);
  *reinterpret_cast<uint2*>(p) =
      make_uint2((uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16),
                 (uint32_t)__bfloat16_as_ushort(c) | ((uint32_t)__bfloat16_as_ushort(e) << 16));
}

template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_kernel(const float* __restrict__ H, int d,
                                                      const int32_t* rows, const int32_t* count, int n,
                                                      const float* __restrict__ gamma, float eps,
                                                      T* __restrict__ xn, T* __restrict__ xn_lo,
                                                      const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int m = count ? *count : n;
  const int j = blockIdx.x;
  if (j >= m) return;
  const int i = rows ? rows[j] : j;
  __shared__ float red[32];
  const float* h = H + (size_t)i * d;
  T* o = xn + (size_t)j * d;
  T* olo = xn_lo ? xn_lo + (size_t)j * d : nullptr;
  constexpr int R = 8;   // float4 of the row per thread: rows up to 8192 stay in registers
  if (d <= 256 * 4 * R) {
    float4 x[R];
    float ss = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int e = (threadIdx.x + r * 256) * 4;
      x[r] = e < d ? *reinterpret_cast<const float4*>(h + e) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) ss += x[r].x * x[r].x + x[r].y * x[r].y + x[r].z * x[r].z + x[r].w * x[r].w;
    ss = block_sum_256(ss, red);
    const float inv = rsqrtf(ss / (float)d + eps);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int e = (threadIdx.x + r * 256) * 4;
      if (e >= d) break;
      const float4 g = *reinterpret_cast<const float4*>(gamma + e);
      const float y[4] = {x[r].x * inv * g.x, x[r].y * inv * g.y, x[r].z * inv * g.z, x[r].w * inv * g.w};
      store4(o + e, y);
      if (olo) {   // remainder term (split activations)
        const float z[4] = {y[0] - to_f(from_f<T>(y[0])), y[1] - to_f(from_f<T>(y[1])),
                            y[2] - to_f(from_f<T>(y[2])), y[3] - to_f(from_f<T>(y[3]))};
        store4(olo + e, z);
      }
    }
    return;
  }
  float ss = 0.f;
  for (int e = threadIdx.x * 4; e < d; e += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(h + e);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = block_sum_256(ss, red);
  const float inv = rsqrtf(ss / (float)d + eps);
  for (int e = threadIdx.x * 4; e < d; e += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(h + e);
    const float4 g = *reinterpret_cast<const float4*>(gamma + e);
    const float y[4] = {v.x * inv * g.x, v.y * inv * g.y, v.z * inv * g.z, v.w * inv * g.w};
    store4(o + e, y);
    if (olo) {
      const float z[4] = {y[0] - to_f(from_f<T>(y[0])), y[1] - to_f(from_f<T>(y[1])),
                          y[2] - to_f(from_f<T>(y[2])), y[3] - to_f(from_f<T>(y[3]))};
      store4(olo + e, z);
    }
  }
}

void launch_rmsnorm(const Ctx& c, const float* H, RowSel sel, const float* gamma, void* xn, void* xn_lo,
                    cudaStream_t s) {
  if (c.dtype == BUDDY_DTYPE_BF16)
    launch_k(rmsnorm_kernel<bf16>, sel.n, 256, 0, s, c.pdl, H, c.d, sel.rows, sel.count, sel.n, gamma,
             c.cfg.rms_eps, (bf16*)xn, (bf16*)xn_lo, (const int32_t*)c.status);
  else
    launch_k(rmsnorm_kernel<float>, sel.n, 256, 0, s, c.pdl, H, c.d, sel.rows, sel.count, sel.n, gamma,
             c.cfg.rms_eps, (float*)xn, (float*)nullptr, (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// QKV finalisation for one layer: bias, rotate-half RoPE at position len[i],
// q kept in fp32, K/V stored (config dtype) at position len[i] of the cache,
// and for the first layer the pooled-context running sum += stored V.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) qkv_finalize_kernel(
    const float* __restrict__ qkv, const float* __restrict__ bias, const int32_t* rows,
    const int32_t* count, int n, int nq, int nkv, int hd, const float* __restrict__ rc,
    const float* __restrict__ rs, const int32_t* len, const int32_t* cache_len, const int64_t* seq_off,
    const int32_t* cap, T* Kc, T* Vc, float* __restrict__ q_out, float* pool, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int m = count ? *count : n;
  const int j = blockIdx.x;
  if (j >= m) return;
  const int i = rows ? rows[j] : j;
  const int pos = len[i];          // RoPE position of the token
  const int cpos = cache_len[i];   // where the layer's cache stores it
  const int half = hd / 2;
  const int N = (nq + 2 * nkv) * hd;
  const float* x = qkv + (size_t)j * N;
  const float* cr = rc + (size_t)pos * half;
  const float* sr = rs + (size_t)pos * half;
  for (int t = threadIdx.x; t < (nq + nkv) * half; t += blockDim.x) {
    const int head = t / half, e = t - head * half;
    const int c0 = head * hd + e;
    float x1 = x[c0], x2 = x[c0 + half];
    if (bias) {
      x1 += bias[c0];
      x2 += bias[c0 + half];
    }
    const float co = cr[e], si = sr[e];
    const float y1 = x1 * co - x2 * si;
    const float y2 = x2 * co + x1 * si;
    if (head < nq) {
      q_out[(size_t)j * nq * hd + c0] = y1;
      q_out[(size_t)j * nq * hd + c0 + half] = y2;
    } else {
      const int g = head - nq;
      T* kp = Kc + kv_offset(seq_off, cap, i, nkv, hd, g, cpos);
      kp[e] = from_f<T>(y1);
      kp[e + half] = from_f<T>(y2);
    }
  }
  const int vbase = (nq + nkv) * hd;
  for (int t = threadIdx.x; t < nkv * hd; t += blockDim.x) {
    const int g = t / hd, e = t - g * hd;
    float v = x[vbase + t];
    if (bias) v += bias[vbase + t];
    const T vs = from_f<T>(v);
    Vc[kv_offset(seq_off, cap, i, nkv, hd, g, cpos) + e] = vs;
    if (pool) pool[(size_t)i * nkv * hd + t] += to_f(vs);
  }
}

void launch_qkv_finalize(const Ctx& c, const float* qkv, const float* bias, RowSel sel,
                         const buddy_kv_state& kv, int layer, float* q_out, float* pool,
                         cudaStream_t s) {
  const int32_t* cl = cache_len(c, kv, layer);
  if (c.dtype == BUDDY_DTYPE_BF16)
    launch_k(qkv_finalize_kernel<bf16>, sel.n, 256, 0, s, c.pdl,
             qkv, bias, sel.rows, sel.count, sel.n, c.nq, c.nkv, c.hd, (const float*)c.rope_cos,
             (const float*)c.rope_sin, (const int32_t*)kv.len, cl, kv.seq_off, kv.cap, (bf16*)kv.k_cache[layer],
             (bf16*)kv.v_cache[layer], q_out, pool, (const int32_t*)c.status);
  else
    launch_k(qkv_finalize_kernel<float>, sel.n, 256, 0, s, c.pdl,
             qkv, bias, sel.rows, sel.count, sel.n, c.nq, c.nkv, c.hd, (const float*)c.rope_cos,
             (const float*)c.rope_sin, (const int32_t*)kv.len, cl, kv.seq_off, kv.cap, (float*)kv.k_cache[layer],
             (float*)kv.v_cache[layer], q_out, pool, (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// Pooled context update for the K and K + V planner features (Sec. 4.3,
// Sec. 5.4): pool[i] += feature of the entry the context layer just stored at
// position pos[i].  (The V feature is added in the QKV epilogue itself.)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) pool_update_kernel(int B, int nkv, int hd, int feature,
                                                          const int32_t* pos, const int64_t* seq_off,
                                                          const int32_t* cap, const T* Kc, const T* Vc,
                                                          float* pool, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int i = blockIdx.y;
  const int x = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B || x >= nkv * hd) return;
  const int g = x / hd, e = x - g * hd;
  const int64_t off = kv_offset(seq_off, cap, i, nkv, hd, g, pos[i]) + e;
  float f = 0.f;
  if (feature != BUDDY_FEATURE_V) f += to_f(Kc[off]);
  if (feature != BUDDY_FEATURE_K) f += to_f(Vc[off]);
  pool[(size_t)i * nkv * hd + x] += f;
}

void launch_pool_update(const Ctx& c, int B, const buddy_kv_state& kv, cudaStream_t s) {
  const int l = c.cl;
  dim3 g((c.kvd + 255) / 256, B);
  if (c.dtype == BUDDY_DTYPE_BF16)
    launch_k(pool_update_kernel<bf16>, g, 256, 0, s, c.pdl, B, c.nkv, c.hd, c.feature, cache_len(c, kv, l),
             kv.seq_off, kv.cap, (const bf16*)kv.k_cache[l], (const bf16*)kv.v_cache[l], kv.pool_sum,
             (const int32_t*)c.status);
  else
    launch_k(pool_update_kernel<float>, g, 256, 0, s, c.pdl, B, c.nkv, c.hd, c.feature, cache_len(c, kv, l),
             kv.seq_off, kv.cap, (const float*)kv.k_cache[l], (const float*)kv.v_cache[l], kv.pool_sum,
             (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// Router, part 1 (Sec. 4.3 + App. C.1 first linear layer):
//   x_i = [ pool_sum[i] / (len[i] + len_bias), expanded over query heads ; h1[i] ]
//   z[i][unit] = W1[unit] . x_i       (bias and SiLU follow in part 2)
// for the Decision Module's r hidden units and, after them, the Budget
// Predictor's rp hidden units (same input, Sec. 4.4); z has r + rp columns.
// Small batches: one CTA per hidden unit and up to 8 sequences; its 8 warps
// take 8 contiguous slices of the 2d-long dot product (four float4 loads of
// W1 in flight per lane), then reduce through shared memory.  Larger batches
// (route_hidden_tiled_kernel): a tiled fp32 GEMM whose K splits leave
// partial sums that part 2 adds in split order.
// ---------------------------------------------------------------------------
constexpr int kRouteRows = 8;
constexpr int kRouteTiledMin = 16;    // batches above this take the tiled router GEMM
constexpr int kRtBM = 64, kRtBN = 64, kRtBK = 32;

__global__ void __launch_bounds__(256) route_hidden_kernel(
    int B, int d, int hd, int group, int nkv, const float* __restrict__ h1,
    const float* __restrict__ pool, const int32_t* len, int len_bias, const float* __restrict__ w1,
    const float* __restrict__ b1, int r, const float* __restrict__ pw1, const float* __restrict__ pb1, int rp,
    float* __restrict__ u, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  __shared__ float red[8][kRouteRows];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int unit = blockIdx.x;
  const int i0 = blockIdx.y * kRouteRows;
  const int nr = min(kRouteRows, B - i0);
  float inv[kRouteRows];
#pragma unroll
  for (int t = 0; t < kRouteRows; ++t) inv[t] = (t < nr) ? 1.0f / (float)(len[i0 + t] + len_bias) : 0.f;
  float acc[kRouteRows];
#pragma unroll
  for (int t = 0; t < kRouteRows; ++t) acc[t] = 0.f;
  const float* wr = unit < r ? w1 + (size_t)unit * 2 * d : pw1 + (size_t)(unit - r) * 2 * d;
  const int kvd = nkv * hd;
  const int per = ((2 * d + 7) / 8 + 3) & ~3;   // elements of a warp's slice (multiple of 4)
  const int k0 = warp * per, k1 = min(2 * d, k0 + per);
#pragma unroll 4
  for (int k = k0 + lane * 4; k < k1; k += 128) {
    const float4 w = __ldg(reinterpret_cast<const float4*>(wr + k));
    if (k < d) {   // pooled half: x[k] = pool[(k / hd) / group * hd + k % hd] / n
      const int qh = k / hd, e = k - qh * hd;
      const int pk = (qh / group) * hd + e;
#pragma unroll
      for (int t = 0; t < kRouteRows; ++t) {
        if (t < nr) {
          const float4 pv = *reinterpret_cast<const float4*>(pool + (size_t)(i0 + t) * kvd + pk);
          acc[t] += (w.x * pv.x + w.y * pv.y + w.z * pv.z + w.w * pv.w) * inv[t];
        }
      }
    } else {
#pragma unroll
      for (int t = 0; t < kRouteRows; ++t) {
        if (t < nr) {
          const float4 hv = *reinterpret_cast<const float4*>(h1 + (size_t)(i0 + t) * d + (k - d));
          acc[t] += w.x * hv.x + w.y * hv.y + w.z * hv.z + w.w * hv.w;
        }
      }
    }
  }
#pragma unroll
  for (int t = 0; t < kRouteRows; ++t) acc[t] = warp_sum(acc[t]);
  if (lane == 0) {
#pragma unroll
    for (int t = 0; t < kRouteRows; ++t) red[warp][t] = acc[t];
  }
  __syncthreads();
  if (threadIdx.x < nr) {
    const int t = threadIdx.x;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) v += red[w][t];
    u[(size_t)(i0 + t) * (r + rp) + unit] = v;
  }
}

// Router part 1 for larger batches, step 1: the router input of every row,
// X[i] = [pool_sum[i] / (len[i] + len_bias) expanded over query heads ; h1[i]]
// ([B, 2d] fp32), so that the GEMM below reads plain rows.
__global__ void __launch_bounds__(256) route_pack_kernel(int d, int hd, int group, int nkv,
                                                         const float* __restrict__ h1,
                                                         const float* __restrict__ pool, const int32_t* len,
                                                         int len_bias, float* __restrict__ X,
                                                         const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int i = blockIdx.x;
  const float inv = 1.0f / (float)(len[i] + len_bias);
  const int kvd = nkv * hd;
  float4* xo = reinterpret_cast<float4*>(X + (size_t)i * 2 * d);
  for (int k = threadIdx.x * 4; k < 2 * d; k += blockDim.x * 4) {
    float4 v;
    if (k < d) {
      const int qh = k / hd, e = k - qh * hd;
      v = *reinterpret_cast<const float4*>(pool + (size_t)i * kvd + (qh / group) * hd + e);
      v.x *= inv; v.y *= inv; v.z *= inv; v.w *= inv;
    } else {
      v = *reinterpret_cast<const float4*>(h1 + (size_t)i * d + (k - d));
    }
    xo[k >> 2] = v;
  }
}

// Router part 1 for larger batches, step 2: Z[i][unit] = X[i] . W[unit] over
// one K split.  Tiles of 64 rows x 64 units, K in steps of 32 staged in
// shared memory (transposed: the inner loop reads 4 consecutive rows and 4
// consecutive units as float4) with the next step's float4 loads in
// registers while the current one is consumed; each of the 256 threads
// accumulates 4 rows x 4 units.  Split s writes slot s of z ([splits, B,
// r + rp]); part 2 adds the slots in split order.
__global__ void __launch_bounds__(256) route_gemm_kernel(int B, int K2, const float* __restrict__ X,
                                                         const float* __restrict__ w1, int r,
                                                         const float* __restrict__ pw1, int rp, int k_per_split,
                                                         float* __restrict__ z, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  __shared__ __align__(16) float xs[kRtBK][kRtBM + 4];
  __shared__ __align__(16) float ws[kRtBK][kRtBN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int u0 = blockIdx.x * kRtBN, i0 = blockIdx.y * kRtBM;
  const int cols = r + rp;
  const int ka = blockIdx.z * k_per_split, kb = min(K2, ka + k_per_split);
  // this thread's two float4 of each tile: (row or unit) = e / 8, k4 = e % 8
  float4 xr[2], wr[2];
  auto fetch = [&](int k0) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int e = tid + q * 256, rr = e >> 3, k = k0 + (e & 7) * 4;
      const int i = i0 + rr, unit = u0 + rr;
      xr[q] = (i < B && k < kb) ? *reinterpret_cast<const float4*>(X + (size_t)i * K2 + k)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
      const float* wp = unit < r ? w1 + (size_t)unit * K2 : pw1 + (size_t)(unit - r) * K2;
      wr[q] = (unit < cols && k < kb) ? __ldg(reinterpret_cast<const float4*>(wp + k))
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  auto stash = [&]() {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int e = tid + q * 256, rr = e >> 3, kk = (e & 7) * 4;
      xs[kk][rr] = xr[q].x; xs[kk + 1][rr] = xr[q].y; xs[kk + 2][rr] = xr[q].z; xs[kk + 3][rr] = xr[q].w;
      ws[kk][rr] = wr[q].x; ws[kk + 1][rr] = wr[q].y; ws[kk + 2][rr] = wr[q].z; ws[kk + 3][rr] = wr[q].w;
    }
  };
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a) acc[a][0] = acc[a][1] = acc[a][2] = acc[a][3] = 0.f;
  fetch(ka);
  for (int k0 = ka; k0 < kb; k0 += kRtBK) {
    __syncthreads();   // the previous step's tiles are consumed
    stash();
    __syncthreads();
    if (k0 + kRtBK < kb) fetch(k0 + kRtBK);   // in flight while this step computes
#pragma unroll 8
    for (int kk = 0; kk < kRtBK; ++kk) {
      const float4 a = *reinterpret_cast<const float4*>(&xs[kk][ty * 4]);
      const float4 b = *reinterpret_cast<const float4*>(&ws[kk][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] += av[p] * bv[q];
    }
  }
  float* zs = z + (size_t)blockIdx.z * B * cols;
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const int i = i0 + ty * 4 + p;
    if (i >= B) continue;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int unit = u0 + tx * 4 + q;
      if (unit < cols) zs[(size_t)i * cols + unit] = acc[p][q];
    }
  }
}

// Router, part 2: s' = W2 u + b2 + omega p~ over the Lm routed layers
// first .. first + Lm - 1, then the deterministic top-k (Eq. 2): layer l is
// selected iff fewer than k_i layers rank above it, where l' ranks above l
// when s'[l'] > s'[l], or s'[l'] == s'[l] and l' < l.  A budget k_i = 0 takes
// the Budget Predictor's k^ = 1 + argmax of its logits (ties to the smaller
// k, Sec. 4.4).  Layers below `first` and the last layer are always set in
// the mask.  One CTA per sequence; a warp per scored layer (and predictor
// logit), its lanes splitting the dot product (eight loads in flight).
__global__ void __launch_bounds__(1024) route_select_kernel(
    int Lm, int first, int r, int rp, const float* __restrict__ z, int splits, int B, const float* __restrict__ b1,
    const float* __restrict__ w2, const float* __restrict__ b2, const float* __restrict__ prior, float omega,
    const float* __restrict__ pb1, const float* __restrict__ pw2, const float* __restrict__ pb2, const int32_t* k,
    uint8_t* mask, int32_t* sel, float* scores, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int i = blockIdx.x;
  extern __shared__ float s[];           // [Lm] scores, [Lm] predictor logits, [r + rp] hidden units
  __shared__ int flag[kMaxLayers];
  __shared__ int kpred;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  float* ui = s + 2 * Lm;
  // hidden units: K-split partial sums in split order, bias, SiLU
  for (int c = threadIdx.x; c < r + rp; c += blockDim.x) {
    float v = 0.f;
    for (int sp = 0; sp < splits; ++sp) v += z[((size_t)sp * B + i) * (r + rp) + c];
    ui[c] = silu_f(v + (c < r ? b1[c] : pb1[c - r]));
  }
  __syncthreads();
  const int ki0 = k[i];
  const bool predict = ki0 == 0 && pw2 != nullptr;
  for (int l = warp; l < (predict ? 2 * Lm : Lm); l += nw) {
    const bool pl = l >= Lm;
    const int row = pl ? l - Lm : l;
    const float* w = pl ? pw2 + (size_t)row * rp : w2 + (size_t)row * r;
    const float* x = pl ? ui + r : ui;
    const int n = pl ? rp : r;
    float a = 0.f;
#pragma unroll 8
    for (int t = lane; t < n; t += 32) a += __ldg(w + t) * x[t];
    a = warp_sum(a);
    if (lane == 0) {
      if (pl) {
        s[l] = a + pb2[row];
      } else {
        a += b2[row];
        if (prior) a += omega * prior[row];
        s[l] = a;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int best = 0;
    if (predict)
      for (int t = 1; t < Lm; ++t)
        if (s[Lm + t] > s[Lm + best]) best = t;
    kpred = predict ? best + 1 : ki0;
  }
  __syncthreads();
  const int ki = kpred;
  for (int l = threadIdx.x; l < Lm; l += blockDim.x) {
    int rank = 0;
    const float v = s[l];
    for (int t = 0; t < Lm; ++t) rank += (s[t] > v) || (s[t] == v && t < l);
    flag[l] = rank < ki;
  }
  __syncthreads();
  const int L = Lm + first + 1;
  for (int l = threadIdx.x; l < Lm; l += blockDim.x) {
    if (scores) scores[(size_t)i * Lm + l] = s[l];
    if (mask) mask[(size_t)i * L + first + l] = (uint8_t)flag[l];
    if (sel) {
      int before = 0;
      for (int t = 0; t < l; ++t) before += flag[t];
      if (flag[l]) sel[(size_t)i * Lm + before] = first + l;
      if (l >= ki) sel[(size_t)i * Lm + l] = -1;
    }
  }
  if (mask)
    for (int l = threadIdx.x; l < first; l += blockDim.x) mask[(size_t)i * L + l] = 1;
  if (threadIdx.x == 0 && mask) mask[(size_t)i * L + L - 1] = 1;
}

// K splits of the tiled router GEMM: about 256 CTAs, at most kRouteZSlots.
static int route_splits(const Ctx& c, int B) {
  if (B <= kRouteTiledMin) return 1;
  const int cols = c.r + (c.have_pred ? c.pred.hidden : 0);
  const int tiles = ((cols + kRtBN - 1) / kRtBN) * ((B + kRtBM - 1) / kRtBM);
  return std::max(1, std::min(kRouteZSlots, 256 / std::max(1, tiles)));
}

void launch_route(const Ctx& c, int B, const float* h1, const float* pool, const int32_t* len,
                  int len_bias, const int32_t* k, uint8_t* mask, int32_t* sel, float* scores,
                  cudaStream_t s) {
  const int rp = c.have_pred ? c.pred.hidden : 0;
  const int cols = c.r + rp;
  const int splits = route_splits(c, B);
  if (B <= kRouteTiledMin) {
    dim3 g1(cols, (B + kRouteRows - 1) / kRouteRows);
    launch_k(route_hidden_kernel, g1, 256, 0, s, c.pdl, B, c.d, c.hd, c.nq / c.nkv, c.nkv, h1, pool, len,
             len_bias, c.dm.w1, c.dm.b1, c.r, c.have_pred ? c.pred.w1 : nullptr, c.have_pred ? c.pred.b1 : nullptr,
             rp, c.dm_u, (const int32_t*)c.status);
  } else {
    launch_k(route_pack_kernel, B, 256, 0, s, c.pdl, c.d, c.hd, c.nq / c.nkv, c.nkv, h1, pool, len, len_bias,
             c.dm_x, (const int32_t*)c.status);
    const int kps = ((2 * c.d + splits - 1) / splits + kRtBK - 1) / kRtBK * kRtBK;
    dim3 g1((cols + kRtBN - 1) / kRtBN, (B + kRtBM - 1) / kRtBM, splits);
    launch_k(route_gemm_kernel, g1, 256, 0, s, c.pdl, B, 2 * c.d, (const float*)c.dm_x, c.dm.w1, c.r,
             c.have_pred ? c.pred.w1 : nullptr, rp, kps, c.dm_u, (const int32_t*)c.status);
  }
  const int sel_threads = 32 * std::min(32, (c.have_pred ? 2 : 1) * c.Lm);
  launch_k(route_select_kernel, B, sel_threads, (2 * c.Lm + cols) * sizeof(float), s, c.pdl, c.Lm, c.cl + 1, c.r,
           rp, (const float*)c.dm_u, splits, B, c.dm.b1, c.dm.w2, c.dm.b2, c.dm.prior, c.dm.omega,
           c.have_pred ? c.pred.b1 : nullptr, c.have_pred ? c.pred.w2 : nullptr,
           c.have_pred ? c.pred.b2 : nullptr, k, mask, sel, scores, (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// Grouping by mask (App. C.1): per layer, the ascending list of sequences that
// execute it and their number (exclusive prefix sum over the mask column).
// Sequences that skip a middle layer get zero K and V at their new position
// in that layer (Sec. 6).  One CTA per layer.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(1024) compact_kernel(int B, int L, int nkv, int hd,
                                                       const uint8_t* __restrict__ mask,
                                                       LayerPtrs ptrs, const int32_t* len,
                                                       const int64_t* seq_off, const int32_t* cap,
                                                       int32_t* rows, int32_t* count, int zero_fill,
                                                       const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int l = blockIdx.x;
  int32_t* rl = rows + (size_t)l * B;
  __shared__ int wsum[32];
  __shared__ int carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int base = 0; base < B; base += blockDim.x) {
    const int i = base + threadIdx.x;
    const int f = (i < B) ? mask[(size_t)i * L + l] : 0;
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    const int before_in_warp = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) wsum[warp] = __popc(bal);
    __syncthreads();
    int before_warps = 0;
    for (int w = 0; w < warp; ++w) before_warps += wsum[w];
    if (f) rl[carry + before_warps + before_in_warp] = i;
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int w = 0; w < nw; ++w) tot += wsum[w];
      carry += tot;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) count[l] = carry;
  // zero K/V at the new position for sequences that skip this layer (the
  // masked variant stores nothing)
  if (!zero_fill || l == 0 || l == L - 1) return;
  T* Kc = (T*)ptrs.k[l];
  T* Vc = (T*)ptrs.v[l];
  const int kvd = nkv * hd;
  for (int i = 0; i < B; ++i) {
    if (mask[(size_t)i * L + l]) continue;
    const int pos = len[i];
    for (int t = threadIdx.x; t < kvd; t += blockDim.x) {
      const int g = t / hd, e = t - g * hd;
      const int64_t off = kv_offset(seq_off, cap, i, nkv, hd, g, pos) + e;
      Kc[off] = from_f<T>(0.f);
      Vc[off] = from_f<T>(0.f);
    }
  }
}

void launch_compact(const Ctx& c, int B, const uint8_t* mask, const buddy_kv_state& kv,
                    int32_t* rows, int32_t* count, cudaStream_t s) {
  LayerPtrs p;
  for (int l = 0; l < c.L; ++l) {
    p.k[l] = kv.k_cache[l];
    p.v[l] = kv.v_cache[l];
  }
  if (c.dtype == BUDDY_DTYPE_BF16)
    launch_k(compact_kernel<bf16>, c.L, 1024, 0, s, c.pdl, B, c.L, c.nkv, c.hd, mask, p,
             (const int32_t*)kv.len, kv.seq_off, kv.cap, rows, count, c.masked ? 0 : 1, (const int32_t*)c.status);
  else
    launch_k(compact_kernel<float>, c.L, 1024, 0, s, c.pdl, B, c.L, c.nkv, c.hd, mask, p,
             (const int32_t*)kv.len, kv.seq_off, kv.cap, rows, count, c.masked ? 0 : 1, (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// Position advance: len[i] += by  (for i < B, or for the listed sequences);
// with a mask (decode step, masked variant) also layer_len[l][i] += mask[i][l].
// ---------------------------------------------------------------------------
__global__ void advance_kernel(int B, int32_t* len, int by, const int32_t* ids, const uint8_t* mask, int L,
                               int32_t* layer_len, int kv_batch, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= B) return;
  const int i = ids ? ids[t] : t;
  len[i] += by;
  if (mask != nullptr)
    for (int l = 0; l < L; ++l) layer_len[(size_t)l * kv_batch + i] += mask[(size_t)t * L + l];
}

void launch_advance(const Ctx& c, int B, int32_t* len, int by, const int32_t* ids, cudaStream_t s,
                    const uint8_t* mask, int32_t* layer_len, int kv_batch) {
  launch_k(advance_kernel, (B + 255) / 256, 256, 0, s, c.pdl, B, len, by, ids, mask, c.L, layer_len, kv_batch,
           (const int32_t*)c.status);
}

// ---------------------------------------------------------------------------
// Prefill / bulk append of positions to one layer (Eq. 9), and the full
// recomputation of the pooled first-layer context for the appended sequences.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) kv_append_kernel(int n_new, int nkv, int hd,
                                                        const int32_t* ids, const int32_t* len,
                                                        const int64_t* seq_off, const int32_t* cap,
                                                        const T* __restrict__ kn,
                                                        const T* __restrict__ vn, T* Kc, T* Vc,
                                                        const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int t = blockIdx.x, jj = blockIdx.y;
  const int s = ids[jj];
  const int pos = len[s] + t;
  const int kvd = nkv * hd;
  const size_t src = ((size_t)jj * n_new + t) * kvd;
  for (int x = threadIdx.x; x < kvd; x += blockDim.x) {
    const int g = x / hd, e = x - g * hd;
    const int64_t off = kv_offset(seq_off, cap, s, nkv, hd, g, pos) + e;
    Kc[off] = kn[src + x];
    Vc[off] = vn[src + x];
  }
}

template <typename T>
__global__ void __launch_bounds__(256) pool_refresh_kernel(int n_new, const int32_t* n_new_of, int nkv, int hd,
                                                           int feature, const int32_t* ids, const int32_t* len,
                                                           const int64_t* seq_off,
                                                           const int32_t* cap, const T* K0, const T* V0,
                                                           float* pool, const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int s = ids ? ids[blockIdx.y] : blockIdx.y;
  const int kvd = nkv * hd;
  const int x = blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= kvd) return;
  const int g = x / hd, e = x - g * hd;
  const int n = len[s] + (n_new_of ? n_new_of[s] : n_new);
  const int64_t off = kv_offset(seq_off, cap, s, nkv, hd, g, 0) + e;
  float acc = 0.f;
  for (int p = 0; p < n; ++p) {
    float f = 0.f;
    if (feature != BUDDY_FEATURE_V) f += to_f(K0[off + (size_t)p * hd]);
    if (feature != BUDDY_FEATURE_K) f += to_f(V0[off + (size_t)p * hd]);
    acc += f;
  }
  pool[(size_t)s * kvd + x] = acc;
}

void launch_kv_append(const Ctx& c, const buddy_kv_state& kv, int layer, int n_seq,
                      const int32_t* ids, int n_new, const void* kn, const void* vn, cudaStream_t s) {
  dim3 g(n_new, n_seq);
  const int32_t* base = cache_len(c, kv, layer);
  if (c.dtype == BUDDY_DTYPE_BF16)
    kv_append_kernel<bf16><<<g, 256, 0, s>>>(n_new, c.nkv, c.hd, ids, base, kv.seq_off, kv.cap,
                                             (const bf16*)kn, (const bf16*)vn,
                                             (bf16*)kv.k_cache[layer], (bf16*)kv.v_cache[layer],
                                             c.status);
  else
    kv_append_kernel<float><<<g, 256, 0, s>>>(n_new, c.nkv, c.hd, ids, base, kv.seq_off, kv.cap,
                                              (const float*)kn, (const float*)vn,
                                              (float*)kv.k_cache[layer], (float*)kv.v_cache[layer],
                                              c.status);
}

void launch_pool_refresh(const Ctx& c, const buddy_kv_state& kv, int n_seq, const int32_t* ids,
                         int n_new, cudaStream_t s) {
  dim3 g((c.kvd + 255) / 256, n_seq);
  const int l = c.cl;
  const int32_t* base = cache_len(c, kv, l);
  if (c.dtype == BUDDY_DTYPE_BF16)
    pool_refresh_kernel<bf16><<<g, 256, 0, s>>>(n_new, nullptr, c.nkv, c.hd, c.feature, ids, base, kv.seq_off,
                                                kv.cap, (const bf16*)kv.k_cache[l], (const bf16*)kv.v_cache[l],
                                                kv.pool_sum, c.status);
  else
    pool_refresh_kernel<float><<<g, 256, 0, s>>>(n_new, nullptr, c.nkv, c.hd, c.feature, ids, base, kv.seq_off,
                                                 kv.cap, (const float*)kv.k_cache[l],
                                                 (const float*)kv.v_cache[l], kv.pool_sum, c.status);
}

// Pooled context of sequences 0..n_seq-1 recomputed over their first
// base + n_new[s] positions of the context layer (prefill).
void launch_pool_refresh_n(const Ctx& c, const buddy_kv_state& kv, int n_seq, const int32_t* n_new,
                           cudaStream_t s) {
  dim3 g((c.kvd + 255) / 256, n_seq);
  const int l = c.cl;
  const int32_t* base = cache_len(c, kv, l);
  if (c.dtype == BUDDY_DTYPE_BF16)
    pool_refresh_kernel<bf16><<<g, 256, 0, s>>>(0, n_new, c.nkv, c.hd, c.feature, nullptr, base, kv.seq_off,
                                                kv.cap, (const bf16*)kv.k_cache[l], (const bf16*)kv.v_cache[l],
                                                kv.pool_sum, c.status);
  else
    pool_refresh_kernel<float><<<g, 256, 0, s>>>(0, n_new, c.nkv, c.hd, c.feature, nullptr, base, kv.seq_off,
                                                 kv.cap, (const float*)kv.k_cache[l],
                                                 (const float*)kv.v_cache[l], kv.pool_sum, c.status);
}

}  // namespace buddy

// Shared device helpers for libbuddy kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/buddy.h"

namespace buddy {

using bf16 = __nv_bfloat16;

// ---------------------------------------------------------------------------
// Element conversions
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

// 8 consecutive elements -> fp32 (16-byte aligned source for bf16, 32 for fp32)
__device__ __forceinline__ void load8(const bf16* p, float* o) {
  uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[2 * i] = __uint_as_float(w[i] << 16);
    o[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void load8(const float* p, float* o) {
  float4 a = __ldg(reinterpret_cast<const float4*>(p));
  float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
  o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + expf(-x)); }

// ---------------------------------------------------------------------------
// Programmatic dependent launch: a kernel launched with programmatic stream
// serialisation may start while its predecessor runs; it must pass pdl_wait()
// before reading anything an earlier kernel wrote.  pdl_trigger() lets the
// next kernel start launching.  Both are no-ops for ordinary launches.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------------------
// Per-call device status: status[0] sticky error bits, status[1] abort flag of
// the call in flight (set by the call's first kernel, read by all others).
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool call_aborted(const int32_t* status) {
  return *reinterpret_cast<const volatile int32_t*>(status + 1) != 0;
}

// Offset (elements) of (sequence i, head g, position p, channel 0) in a cache.
__device__ __forceinline__ int64_t kv_offset(const int64_t* seq_off, const int32_t* cap, int i,
                                             int n_kv, int hd, int g, int p) {
  return ((seq_off[i] * n_kv + (int64_t)g * cap[i] + p) * (int64_t)hd);
}

}  // namespace buddy

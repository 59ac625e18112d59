// buddy_route_noalloc: the router for callers that must not allocate device
// memory (no context, no cudaMalloc).  Its scratch — the call's abort word and
// the Decision Module's hidden activations — lives in one file-scope device
// array that every GPU loading this library holds until the process exits.
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace buddy {

// Route kernels shared with buddy_route (kernels.cu).
__global__ void route_hidden_kernel(int B, int d, int hd, int group, int nkv, const float* h1,
                                    const float* pool, const int32_t* len, int len_bias,
                                    const float* w1, const float* b1, int r, const float* pw1,
                                    const float* pb1, int rp, float* u, const int32_t* status);
__global__ void route_select_kernel(int Lm, int first, int r, int rp, const float* z, int splits, int B,
                                    const float* b1, const float* w2, const float* b2, const float* prior,
                                    float omega, const float* pb1, const float* pw2, const float* pb2,
                                    const int32_t* k, uint8_t* mask, int32_t* sel, float* scores,
                                    const int32_t* status);

// Layout of the static scratch: words [0, 64) hold status (word 1 = abort
// flag of the call in flight), then batch * dm_hidden fp32 hidden units.
constexpr int kNoAllocHeader = 64;
constexpr int kNoAllocMaxUnits = 65536;   // batch * dm_hidden (256 KiB of fp32)
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocHeader + kNoAllocMaxUnits];

constexpr int kMaxDevices = 64;
static void* g_scratch_addr[kMaxDevices];
static std::mutex g_scratch_mu;

// Checks budgets and lengths for the call, publishes the abort word and the
// caller-visible flags.  Single CTA.
__global__ void noalloc_check_kernel(int B, const int32_t* k, int Lm, const int32_t* len,
                                     int32_t* status, int32_t* flags_out) {
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  int b = 0;
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    const int ki = k[i];
    if (ki < 1 || ki > Lm) b |= BUDDY_DEV_BAD_BUDGET;
    if (len[i] < 1) b |= BUDDY_DEV_BAD_POSITION;
  }
  if (b) atomicOr(&bad, b);
  __syncthreads();
  if (threadIdx.x == 0) {
    status[1] = bad ? 1 : 0;
    if (flags_out) *flags_out = bad;
  }
}

// Device address of the static scratch on the current device, looked up once
// per device (cudaGetSymbolAddress must not run inside a stream capture).
static cudaError_t scratch_address(float** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = static_cast<float*>(g_scratch_addr[dev]);
  return cudaSuccess;
}

}  // namespace buddy

using namespace buddy;

extern "C" int buddy_route_noalloc(int32_t n_layers, int32_t d_model, int32_t n_q_heads,
                                   int32_t n_kv_heads, int32_t head_dim, int32_t dm_hidden,
                                   const buddy_dm_weights* dm, int32_t batch, const float* pool_sum,
                                   const int32_t* len, const float* h1, const int32_t* k,
                                   int32_t* sel_out, uint8_t* mask_out, float* scores_out,
                                   int32_t* flags_out, void* stream) {
  if (!dm || !dm->w1 || !dm->b1 || !dm->w2 || !dm->b2 || !pool_sum || !len || !h1 || !k)
    return BUDDY_ERR_ARG;
  if (n_layers < 3 || n_layers > kMaxLayers || n_q_heads <= 0 || n_kv_heads <= 0 ||
      (head_dim != 64 && head_dim != 128) || n_q_heads % n_kv_heads != 0 ||
      d_model != n_q_heads * head_dim || dm_hidden <= 0 || batch < 1)
    return BUDDY_ERR_ARG;
  if ((int64_t)batch * dm_hidden > kNoAllocMaxUnits) return BUDDY_ERR_RANGE;
  float* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return BUDDY_ERR_CUDA;
  int32_t* status = reinterpret_cast<int32_t*>(scratch);
  float* u = scratch + kNoAllocHeader;
  cudaStream_t s = (cudaStream_t)stream;
  const int Lm = n_layers - 2;
  noalloc_check_kernel<<<1, 256, 0, s>>>(batch, k, Lm, len, status, flags_out);
  dim3 g1(dm_hidden, (batch + 7) / 8);
  route_hidden_kernel<<<g1, 256, 0, s>>>(batch, d_model, head_dim, n_q_heads / n_kv_heads, n_kv_heads,
                                         h1, pool_sum, len, 0, dm->w1, dm->b1, dm_hidden, nullptr, nullptr, 0,
                                         u, status);
  const int sel_threads = 32 * (Lm < 32 ? Lm : 32);
  route_select_kernel<<<batch, sel_threads, (2 * Lm + dm_hidden) * sizeof(float), s>>>(
      Lm, 1, dm_hidden, 0, u, 1, batch, dm->b1, dm->w2, dm->b2, dm->prior, dm->omega, nullptr, nullptr, nullptr, k,
      mask_out, sel_out, scores_out, status);
  return cudaGetLastError() == cudaSuccess ? BUDDY_OK : BUDDY_ERR_CUDA;
}

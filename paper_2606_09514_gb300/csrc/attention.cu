// Decode attention for one layer (Eq. 9): for every active row j (sequence
// i = rows[j]) and KV head g, the G = n_q / n_kv query heads of the group
// attend over positions 0..len[i] of that head's cache (the new token included;
// zero-filled positions of earlier skipped steps take part with logit 0).
//
// Two work loops:
//   * bf16 caches (G <= 8): the tensor-core loop of attn_tc.cuh (warp shares
//     of the concatenated position streams, mma.sync contractions, span
//     partials merged by the warp that completes a stream), or at a few rows
//     the cluster loop of attn_cl.cu;
//   * fp32 caches: the CUDA-core
//     loop of attn_common.cuh.  Its work items are (row, KV head, span of P
//     positions); P is derived on the device from the total number of
//     positions so that there are about as many items as half the grid
//     (64 <= P <= 1024).  Persistent CTAs walk the items.  Inside an item the
//     CTA streams chunks of 64 positions: K and V are copied into shared
//     memory with 16-byte cp.async (double-buffered; K rows padded so that
//     lanes reading 32 different positions hit distinct banks), then logits,
//     an online softmax and P.V run in fp32.  An item covering the whole row
//     writes the output; otherwise it writes a partial (running max, sum of
//     exponentials, unnormalised output) and the last item of the (row, head)
//     to finish merges the partials in span order (log-sum-exp).
#include <cuda_runtime.h>

#include <algorithm>

#include "attn_common.cuh"
#include "attn_tc.cuh"
#include "common.cuh"
#include "internal.h"

namespace buddy {

template <int HD, bool SPLIT>
__global__ void __launch_bounds__(kTcaThreads) attn_tc_kernel(AttnArgs<bf16> A) {
  extern __shared__ __align__(16) uint8_t smraw[];
  __shared__ int sc[4];
  attn_tc_run<HD, SPLIT>(A, blockIdx.x, gridDim.x, smraw, sc, true);
}

// bf16 caches with at most 8 query heads per KV head: the tensor-core loop
template <int HD, bool SPLIT>
static void attn_tc_impl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q, void* out,
                         void* out_lo, cudaStream_t s) {
  const size_t smem = attn_tc_smem_bytes(HD, c.maxB);
  static int occ = 0;   // one per instantiation
  static size_t occ_smem = 0;
  if (occ == 0 || occ_smem != smem) {
    cudaFuncSetAttribute(attn_tc_kernel<HD, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, attn_tc_kernel<HD, SPLIT>, kTcaThreads, smem) !=
        cudaSuccess)
      occ = 1;
    occ_smem = smem;
  }
  const int grid = c.num_sms * std::max(1, std::min(occ, 4));
  AttnArgs<bf16> A{q, sel.rows, sel.count, sel.n, c.nq, c.nkv, cache_len(c, kv, layer), kv.seq_off, kv.cap,
                   (const bf16*)kv.k_cache[layer], (const bf16*)kv.v_cache[layer], c.attn_max_chunks, c.attn_m,
                   c.attn_l, c.attn_acc, c.attn_ctr, (bf16*)out, (bf16*)out_lo, c.status};
  launch_k(attn_tc_kernel<HD, SPLIT>, grid, kTcaThreads, smem, s, c.pdl, A);
}

template <typename T, int HD, int GP>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(AttnArgs<T> A) {
  extern __shared__ __align__(16) uint8_t smraw[];
  __shared__ float sc[32];
  attn_run<T, HD, GP, kAttnThreads>(A, threadIdx.x, blockIdx.x, gridDim.x, smraw, sc, SyncCta{}, true);
}

template <typename T, int HD, int GP>
static void attn_impl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q,
                      void* out, void* out_lo, cudaStream_t s) {
  const int G = c.nq / c.nkv;
  const size_t smem = attn_smem_bytes(attn_smem_fixed<T, HD>(), G, HD, c.attn_max_chunks, c.maxB);
  static bool attr_set = false;   // one per instantiation
  static int occ = 0;
  static size_t occ_smem = 0;
  if (!attr_set) {
    cudaFuncSetAttribute(attn_kernel<T, HD, GP>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    attr_set = true;
  }
  if (occ == 0 || occ_smem != smem) {   // resident CTAs per SM at this shared-memory size
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, attn_kernel<T, HD, GP>, kAttnThreads, smem) !=
        cudaSuccess)
      occ = 1;
    occ_smem = smem;
  }
  const int grid = c.num_sms * std::max(1, std::min(occ, 4));
  AttnArgs<T> A{q, sel.rows, sel.count, sel.n, c.nq, c.nkv, cache_len(c, kv, layer), kv.seq_off, kv.cap,
                (const T*)kv.k_cache[layer], (const T*)kv.v_cache[layer], c.attn_max_chunks, c.attn_m, c.attn_l,
                c.attn_acc, c.attn_ctr, (T*)out, (T*)out_lo, c.status};
  launch_k(attn_kernel<T, HD, GP>, grid, kAttnThreads, smem, s, c.pdl, A);
}

template <typename T, int HD>
static void attn_group(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q, void* out,
                       void* out_lo, cudaStream_t s) {
  switch (attn_group_pad(c.nq / c.nkv)) {
    case 1: attn_impl<T, HD, 1>(c, sel, kv, layer, q, out, out_lo, s); break;
    case 2: attn_impl<T, HD, 2>(c, sel, kv, layer, q, out, out_lo, s); break;
    case 4: attn_impl<T, HD, 4>(c, sel, kv, layer, q, out, out_lo, s); break;
    default: attn_impl<T, HD, 8>(c, sel, kv, layer, q, out, out_lo, s);
  }
}

// Partial slots per (row, query head): the CUDA-core loop's spans are at least
// kChunk positions long; the tensor-core loop's at least kTcaMinShare, plus
// one for a share boundary.
int attention_max_spans(int max_pos) {
  return std::max((max_pos + kChunk - 1) / kChunk, attn_tc_max_spans(max_pos));
}

// bf16 caches with at most 8 query heads per KV head whose per-row tables fit
// next to the chunk buffers take the tensor-core loop
bool attention_tc(const Ctx& c) {
  return c.dtype == BUDDY_DTYPE_BF16 && c.nq / c.nkv <= 8 &&
         attn_tc_smem_bytes(c.hd, c.maxB) <= (size_t)kTcaSmemLimit;
}

void launch_attention(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q,
                      void* out, void* out_lo, cudaStream_t s) {
  if (attention_cl(c)) {
    launch_attention_cl(c, sel, kv, layer, q, out, out_lo, s);
  } else if (attention_tc(c)) {
    if (c.hd == 128) {
      if (out_lo) attn_tc_impl<128, true>(c, sel, kv, layer, q, out, out_lo, s);
      else attn_tc_impl<128, false>(c, sel, kv, layer, q, out, out_lo, s);
    } else {
      if (out_lo) attn_tc_impl<64, true>(c, sel, kv, layer, q, out, out_lo, s);
      else attn_tc_impl<64, false>(c, sel, kv, layer, q, out, out_lo, s);
    }
  } else if (c.dtype == BUDDY_DTYPE_BF16) {
    if (c.hd == 128) attn_group<bf16, 128>(c, sel, kv, layer, q, out, out_lo, s);
    else attn_group<bf16, 64>(c, sel, kv, layer, q, out, out_lo, s);
  } else {
    if (c.hd == 128) attn_group<float, 128>(c, sel, kv, layer, q, out, nullptr, s);
    else attn_group<float, 64>(c, sel, kv, layer, q, out, nullptr, s);
  }
}

}  // namespace buddy

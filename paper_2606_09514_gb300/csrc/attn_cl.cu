// Decode attention for small batches (Eq. 9): one thread-block cluster per
// (active row, KV head) stream, the span merge done inside the cluster.
//
// At a few rows the streams are few (batch 1 of an 8-KV-head model: 8
// streams of ~2k positions) and short: cutting them across the whole GPU
// leaves tens of partial results per stream whose merge costs as much as the
// streaming.  Here a cluster of C CTAs (C = 16 where the device allows it,
// else 8) takes one stream: CTA r streams positions [r np / C, (r+1) np / C)
// with its 4 warps (contiguous quarters, 32-position chunks through a
// 2-buffer cp.async ring per warp; the contractions are those of the
// tensor-core loop in attn_tc.cuh: S^T = K Q^T and O^T += V^T P^T on
// mma.sync m16n8k16 with the G <= 8 query heads as the 8 columns, base-2
// online softmax).  The 4 warps' partials are merged in shared memory and
// every CTA stores its partial into CTA 0's gather area through distributed
// shared memory (st.shared::cluster), cut by output: the G x HD outputs of
// the stream are split into C contiguous slices and CTA s owns slice s.
// Every CTA stores its (m, l) of each head and its unnormalised output of
// each (head, channel) into the gather area of that output's owner; after
// one cluster barrier (release / acquire) every CTA merges the C partials of
// its own slice from its own shared memory (log-sum-exp, in rank order:
// deterministic) and writes those outputs.  No kernel-wide or cross-cluster
// waits; every CTA reaches the cluster barrier (a cluster whose row is past
// the row count leaves before it, all of its CTAs together).
#include <cuda_runtime.h>

#include <algorithm>

#include "attn_tc.cuh"
#include "common.cuh"
#include "internal.h"

namespace buddy {

constexpr int kClWarps = 4;
constexpr int kClThreads = 32 * kClWarps;
constexpr int kClChunk = 32;
constexpr int kClStages = 2;
constexpr int kClMaxCtas = 16;

constexpr int kClMaxStreams = 64;   // (rows x KV heads) up to which the cluster kernel is used

template <int HD>
__host__ __device__ constexpr size_t attn_cl_bufs() {
  // per warp: kClStages buffers of K and V rows (padded by 8 bf16)
  return (size_t)kClWarps * kClStages * 2 * kClChunk * (HD + 8) * 2;
}
// One partial in an owner's gather area: m[8], l[8], then the owner's slice
// of outputs (at most 8 heads x HD channels / 8 CTAs).
template <int HD>
__host__ __device__ constexpr int attn_cl_gstride() {
  return 16 + HD;
}
template <int HD>
__host__ __device__ constexpr size_t attn_cl_smem() {
  // the warps' partials (m, l per head, o per head and channel) reuse the
  // buffers once the streaming is done; then the gather area, one partial
  // per CTA of the cluster
  const size_t parts = (size_t)kClWarps * 8 * (HD + 2) * 4;
  return (attn_cl_bufs<HD>() > parts ? attn_cl_bufs<HD>() : parts) +
         (size_t)kClMaxCtas * attn_cl_gstride<HD>() * 4;
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(r)
               : "r"((uint32_t)__cvta_generic_to_shared(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_dsmem(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_dsmem4(uint32_t addr, const float* v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v[0]), "f"(v[1]), "f"(v[2]),
               "f"(v[3])
               : "memory");
}

template <int HD, bool SPLIT>
__global__ void __launch_bounds__(kClThreads) attn_cl_kernel(AttnArgs<bf16> A) {
  extern __shared__ __align__(16) uint8_t smraw[];
  constexpr int CH = kClChunk, NST = kClStages;
  constexpr int KROW = HD + 8;
  constexpr int KSTEPS = HD / 16;
  constexpr int DT = HD / 8;
  constexpr int V16 = HD / 8;
  constexpr int PSTRIDE = 8 * (HD + 2);   // one partial: m[8], l[8], o[8][HD]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nq = A.nq, nkv = A.nkv, G = nq / nkv;
  const int stream = blockIdx.y;
  const int j = stream / nkv, g = stream - j * nkv;
  // row count and rows were written by the compaction kernel, which completed
  // before this kernel's predecessor let it launch
  const int m = A.count ? *A.count : A.n;
  if (j >= m || call_aborted(A.status)) {   // uniform across the cluster
    pdl_wait();
    pdl_trigger();
    return;
  }
  const uint32_t rank = cluster_rank(), C = cluster_size();
  const int i = A.rows ? A.rows[j] : j;
  const int np = A.len[i] + 1;   // cached positions and the new token
  const int c0 = (int)((int64_t)np * rank / C), c1 = (int)((int64_t)np * (rank + 1) / C);
  const int w0 = c0 + (c1 - c0) * warp / kClWarps, w1 = c0 + (c1 - c0) * (warp + 1) / kClWarps;
  const int64_t kvo = (A.seq_off[i] * nkv + (int64_t)g * A.cap[i]) * HD;
  bf16* wbuf = reinterpret_cast<bf16*>(smraw) + (size_t)warp * NST * 2 * CH * KROW;
  float* parts = reinterpret_cast<float*>(smraw);   // overlays the buffers after the streaming
  float* mine = parts + (size_t)warp * PSTRIDE;
  constexpr int GS = attn_cl_gstride<HD>();
  constexpr size_t kBufBytes = attn_cl_smem<HD>() - (size_t)kClMaxCtas * GS * 4;
  float* gather = reinterpret_cast<float*>(smraw + kBufBytes);   // one partial per CTA of the cluster

  auto issue = [&](int p, int cnt, int buf) {
    bf16* Kd = wbuf + (size_t)buf * 2 * CH * KROW;
    bf16* Vd = Kd + CH * KROW;
    constexpr int RPI = 32 / V16;
    const int pl = lane / V16, sl = lane % V16;
    const bf16* ks = A.Kc + kvo + (int64_t)p * HD + pl * HD + sl * 8;
    const bf16* vs = A.Vc + kvo + (int64_t)p * HD + pl * HD + sl * 8;
    const int so = pl * KROW + sl * 8;
#pragma unroll 4
    for (int r = 0; r + pl < cnt; r += RPI) {
      cp_async16(Kd + so + r * KROW, ks + (size_t)r * HD);
      cp_async16(Vd + so + r * KROW, vs + (size_t)r * HD);
    }
    for (int x = cnt * V16 + lane; x < CH * V16; x += 32) {   // rows past the chunk: zero V
      const int r = x / V16, q = x - r * V16;
      *reinterpret_cast<uint4*>(Vd + r * KROW + q * 8) = make_uint4(0u, 0u, 0u, 0u);
    }
  };

  // prologue: every cached position may be copied before the wait; only the
  // new token (position np - 1, written by the preceding kernel) comes after
  // it, into the last row of its chunk.  A warp whose whole range fits in its
  // NST buffers loads all of it here (the loop below then issues nothing);
  // otherwise the first NST - 1 chunks, one buffer staying free for the loop.
  const int pre = (w1 - w0 + CH - 1) / CH <= NST ? NST : NST - 1;
  int xi = w0, k0 = 0, late_row = -1, late_buf = 0;
  for (; k0 < pre && xi < w1; ++k0) {
    const int cnt = min(CH, w1 - xi);
    if (xi + cnt == np) {
      issue(xi, cnt - 1, k0);   // also zero-fills V rows cnt - 1 .. CH - 1
      cp_async_commit();
      late_row = cnt - 1;
      late_buf = k0;
      xi += cnt;
      ++k0;
      break;
    }
    issue(xi, cnt, k0);
    cp_async_commit();
    xi += cnt;
  }
  pdl_wait();
  pdl_trigger();
  if (late_row >= 0) {
    __syncwarp();   // the zero fill of that row is done before the copy lands there
    bf16* Kd = wbuf + (size_t)late_buf * 2 * CH * KROW + (size_t)late_row * KROW;
    bf16* Vd = Kd + CH * KROW;
    const bf16* ks = A.Kc + kvo + (int64_t)(np - 1) * HD;
    const bf16* vs = A.Vc + kvo + (int64_t)(np - 1) * HD;
    for (int x = lane; x < V16; x += 32) {
      cp_async16(Kd + x * 8, ks + x * 8);
      cp_async16(Vd + x * 8, vs + x * 8);
    }
    cp_async_commit();
  }
  for (int k = k0; k < NST - 1; ++k) {
    if (xi < w1) {
      const int cnt = min(CH, w1 - xi);
      issue(xi, cnt, k);
      xi += cnt;
    }
    cp_async_commit();
  }

  // queries of the group as the B operand (column = head h0 < G, rows = dims)
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);   // log2(e) / sqrt(d_h)
  const int h0 = lane >> 2, c2 = (lane & 3) * 2;
  uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
  {
    const float* qj = A.q + ((size_t)j * nq + (size_t)g * G + h0) * HD;
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
  }
  float mrun[2] = {-INFINITY, -INFINITY}, lrun[2] = {0.f, 0.f};
  float o[DT / 2][4];
#pragma unroll
  for (int t = 0; t < DT / 2; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;

  for (int xc = w0, k = 0; xc < w1; ++k) {
    if (xi < w1) {
      const int cnt = min(CH, w1 - xi);
      issue(xi, cnt, (k + NST - 1) % NST);
      xi += cnt;
    }
    cp_async_commit();
    const int cnt = min(CH, w1 - xc);
    cp_async_wait<NST - 1>();
    __syncwarp();
    const bf16* Ks = wbuf + (size_t)(k % NST) * 2 * CH * KROW;
    const bf16* Vs = Ks + CH * KROW;
    constexpr int MT = CH / 16;
    float sv[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
      const bf16* kr = Ks + (size_t)(mt * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * KROW + 8 * (lane >> 4);
#pragma unroll
      for (int kk = 0; kk < KSTEPS; ++kk) {
        uint32_t a0, a1, a2, a3;
        tca::ldsm_x4(kr + kk * 16, a0, a1, a2, a3);
        tca::mma16816(acc[kk & 1], a0, a1, a2, a3, qh[kk][0], qh[kk][1]);
        if (SPLIT) tca::mma16816(acc[kk & 1], a0, a1, a2, a3, ql[kk][0], ql[kk][1]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) sv[mt][e] = acc[0][e] + acc[1][e];
    }
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
      alpha[e] = tca::exp2a(mrun[e] - mn);
      mrun[e] = mn;
      ps[e] = 0.f;
    }
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        sv[mt][e] = tca::exp2a(sv[mt][e] - mrun[e & 1]);
        ps[e & 1] += sv[mt][e];
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
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
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
    xc += cnt;
  }
  cp_async_wait<0>();
  __syncthreads();   // every warp is done with its buffers

  // this warp's partial: heads c2 + e (e = 0, 1), channels 16 t + h0 (+ 8)
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int hh = c2 + e;
    if (hh < 8) {
      if (h0 == 0) {
        mine[hh] = mrun[e];
        mine[8 + hh] = lrun[e];
      }
      float* oh = mine + 16 + (size_t)hh * HD;
#pragma unroll
      for (int t = 0; t < DT / 2; ++t) {
        oh[16 * t + h0] = o[t][e];
        oh[16 * t + h0 + 8] = o[t][2 + e];
      }
    }
  }
  __syncthreads();
  // the CTA's partial, the warps' partials merged per (head, channel), stored
  // into the gather area of the output's owner (slot `rank`), four channels
  // per thread and per 16-byte store (a slice is a multiple of 4 outputs:
  // G * HD is a multiple of 64 and C is 8 or 16)
  const int SL = (G * HD + (int)C - 1) / (int)C;   // outputs per owner (<= HD for C >= 8)
  for (int x = tid * 4; x < G * HD; x += kClThreads * 4) {
    const int hh = x / HD, ch = x - hh * HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kClWarps; ++w) M = fmaxf(M, parts[w * PSTRIDE + hh]);
    float L = 0.f, Ov[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int w = 0; w < kClWarps; ++w) {
      const float mw = parts[w * PSTRIDE + hh];
      const float f = mw == -INFINITY ? 0.f : tca::exp2a(mw - M);
      L += f * parts[w * PSTRIDE + 8 + hh];
      const float4 pv = *reinterpret_cast<const float4*>(parts + w * PSTRIDE + 16 + hh * HD + ch);
      Ov[0] += f * pv.x;
      Ov[1] += f * pv.y;
      Ov[2] += f * pv.z;
      Ov[3] += f * pv.w;
    }
    const uint32_t own = (uint32_t)(x / SL);
    float* slot = gather + (size_t)rank * GS;
    st_dsmem4(dsmem_addr(slot + 16 + (x - (int)own * SL), own), Ov);
    // (m, l) of head hh to every owner whose slice holds one of its outputs
    if (ch == 0) {
      const uint32_t o1 = (uint32_t)(((hh + 1) * HD - 1) / SL);
      for (uint32_t o = own; o <= o1; ++o) {
        st_dsmem(dsmem_addr(slot + hh, o), M);
        st_dsmem(dsmem_addr(slot + 8 + hh, o), L);
      }
    }
  }
  cluster_sync();   // every partial has landed in its owner's gather area
  const size_t obase = ((size_t)j * nq + (size_t)g * G) * HD;
  const int x0 = (int)rank * SL, x1 = min(G * HD, x0 + SL);
  for (int x = x0 + tid * 4; x < x1; x += kClThreads * 4) {
    const int hh = x / HD;
    float M = -INFINITY;
    for (uint32_t r = 0; r < C; ++r) M = fmaxf(M, gather[r * GS + hh]);
    float L = 0.f, Ov[4] = {0.f, 0.f, 0.f, 0.f};
    for (uint32_t r = 0; r < C; ++r) {
      const float mr = gather[r * GS + hh];
      const float f = mr == -INFINITY ? 0.f : tca::exp2a(mr - M);
      L += f * gather[r * GS + 8 + hh];
      const float4 gv = *reinterpret_cast<const float4*>(gather + r * GS + 16 + (x - x0));
      Ov[0] += f * gv.x;
      Ov[1] += f * gv.y;
      Ov[2] += f * gv.z;
      Ov[3] += f * gv.w;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) store_out(A.out, A.out_lo, obase + (size_t)(x + e), Ov[e] / L);
  }
}

// Clusters of C CTAs the device can hold at once (C = 16 and 8), queried
// once per instantiation; 0 where the size cannot be scheduled.
template <int HD, bool SPLIT>
static const int* cl_capacity() {
  static int cap[2] = {-1, -1};   // [0]: C = 16, [1]: C = 8
  if (cap[0] >= 0) return cap;
  const size_t smem = attn_cl_smem<HD>();
  cudaFuncSetAttribute(attn_cl_kernel<HD, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  for (int v = 0; v < 2; ++v) {
    const int C = v == 0 ? kClMaxCtas : 8;
    cap[v] = 0;
    if (C > 8 && cudaFuncSetAttribute(attn_cl_kernel<HD, SPLIT>, cudaFuncAttributeNonPortableClusterSizeAllowed,
                                      1) != cudaSuccess) {
      cudaGetLastError();
      continue;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C, 1, 1);
    cfg.blockDim = dim3(kClThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_cl_kernel<HD, SPLIT>, &cfg) == cudaSuccess) cap[v] = n;
    cudaGetLastError();
  }
  return cap;
}

// Cluster size for `streams` streams: 16 CTAs when every cluster fits at
// once (a cluster that waits for another to finish doubles the latency),
// else 8; 0 if neither size can be scheduled.
template <int HD, bool SPLIT>
static int cl_size(int streams) {
  const int* cap = cl_capacity<HD, SPLIT>();
  if (cap[0] > 0 && (streams <= cap[0] || cap[1] <= 0)) return kClMaxCtas;
  return cap[1] > 0 ? 8 : 0;
}

bool attention_cl(const Ctx& c) {
  if (!(c.dtype == BUDDY_DTYPE_BF16 && c.nq / c.nkv <= 8 && c.maxB * c.nkv <= kClMaxStreams)) return false;
  return (c.hd == 128 ? cl_size<128, false>(c.maxB * c.nkv) : cl_size<64, false>(c.maxB * c.nkv)) > 0;
}

template <int HD, bool SPLIT>
static void attn_cl_impl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q, void* out,
                         void* out_lo, cudaStream_t s) {
  const int C = cl_size<HD, SPLIT>(sel.n * c.nkv);
  AttnArgs<bf16> A{q, sel.rows, sel.count, sel.n, c.nq, c.nkv, cache_len(c, kv, layer), kv.seq_off, kv.cap,
                   (const bf16*)kv.k_cache[layer], (const bf16*)kv.v_cache[layer], 0, nullptr, nullptr, nullptr,
                   nullptr, (bf16*)out, (bf16*)out_lo, c.status};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C, sel.n * c.nkv, 1);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = attn_cl_smem<HD>();
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = C;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = c.pdl ? 2 : 1;
  cudaLaunchKernelEx(&cfg, attn_cl_kernel<HD, SPLIT>, A);
}

void launch_attention_cl(const Ctx& c, RowSel sel, const buddy_kv_state& kv, int layer, const float* q, void* out,
                         void* out_lo, cudaStream_t s) {
  if (c.hd == 128) {
    if (out_lo) attn_cl_impl<128, true>(c, sel, kv, layer, q, out, out_lo, s);
    else attn_cl_impl<128, false>(c, sel, kv, layer, q, out, out_lo, s);
  } else {
    if (out_lo) attn_cl_impl<64, true>(c, sel, kv, layer, q, out, out_lo, s);
    else attn_cl_impl<64, false>(c, sel, kv, layer, q, out, out_lo, s);
  }
}

}  // namespace buddy

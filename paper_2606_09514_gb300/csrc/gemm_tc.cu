// tcgen05 / TMA GEMM for bf16 decode projections (placeholder until the
// tensor-core path lands; every GEMM currently runs on the CUDA-core kernel).
#include "internal.h"

namespace buddy {

int gemm_tc_prepare(Ctx& c) {
  c.use_tc = false;
  return BUDDY_OK;
}

bool gemm_tc_supported(const Ctx&) { return false; }

void launch_gemm_tc(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s) {
  launch_gemm_simt(c, epi, a, s);
}

}  // namespace buddy

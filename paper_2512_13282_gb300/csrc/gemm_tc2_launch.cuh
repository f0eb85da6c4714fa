// gemm_tc2_launch.cuh -- cluster launch of the CTA-pair kernel (included by
// the instantiation translation units).
#pragma once
#include "gemm_internal.h"
#include "gemm_tc2.cuh"

namespace gb300 {

template <int BN, int STAGES, bool KM, int EPI, int EW, int TMA>
cudaError_t launch_pair(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o, const CUtensorMap &w, const TcParams &p,
                        int grid,
                        cudaStream_t st) {
  using Cfg = Tc2Cfg<BN, STAGES, KM, EPI, EW, TMA>;
  auto kern = gemm_tc2_kernel<BN, STAGES, KM, EPI, EW, TMA>;
  static bool opted_in[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || !opted_in[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) opted_in[dev] = true;
  }
  // grid is even: a whole number of pairs
  return launch_ex(kern, dim3((unsigned)grid), dim3(Cfg::kThreads), Cfg::kSmemBytes, st, 2, a, b, o, w, p);
}

}  // namespace gb300

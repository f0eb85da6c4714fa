// Instantiations of the tcgen05 kernel with the bf16 epilogue.
#include "gemm_internal.h"

namespace gb300 {

namespace {
template <int BN, int STAGES, bool KM, int EPI, int EW>
cudaError_t launch_one(const CUtensorMap &a, const CUtensorMap &b, const TcParams &p, int grid,
                       cudaStream_t st) {
  using Cfg = TcCfg<BN, STAGES, KM, EPI, EW>;
  auto kern = gemm_tc_kernel<BN, STAGES, KM, EPI, EW>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  kern<<<grid, Cfg::kThreads, Cfg::kSmemBytes, st>>>(a, b, p);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_tc_bf16(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const TcParams &p, int grid, cudaStream_t st) {
  if (v.bn == 256)
    return v.b_kmajor ? launch_one<256, 4, true, kEpiBf16, 4>(a, b, p, grid, st)
                      : launch_one<256, 4, false, kEpiBf16, 4>(a, b, p, grid, st);
  return v.b_kmajor ? launch_one<128, 6, true, kEpiBf16, 4>(a, b, p, grid, st)
                    : launch_one<128, 6, false, kEpiBf16, 4>(a, b, p, grid, st);
}

}  // namespace gb300

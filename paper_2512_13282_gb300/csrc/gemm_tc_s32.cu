// Instantiations of the tcgen05 kernel with the exact int32 (slab) epilogue.
#include "gemm_internal.h"

namespace gb300 {

namespace {
template <int BN, int STAGES, bool KM, int EPI, int EW, int TMA>
cudaError_t launch_one(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o, const CUtensorMap &w, const TcParams &p,
                       int grid,
                       cudaStream_t st) {
  using Cfg = TcCfg<BN, STAGES, KM, EPI, EW, TMA>;
  auto kern = gemm_tc_kernel<BN, STAGES, KM, EPI, EW, TMA>;
  // the shared-memory opt-in is per device and kernel: set it once
  static bool opted_in[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || !opted_in[dev]) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) opted_in[dev] = true;
  }
  return launch_ex(kern, dim3((unsigned)grid), dim3(Cfg::kThreads), Cfg::kSmemBytes, st, 1, a, b, o, w, p);
}
}  // namespace

// Tile widths compiled for the int32 epilogue: 128 (one epilogue warpgroup,
// 128 int32 accumulators per thread, 6 stages), 192, 224 (B column-major
// only) and 256 (two warpgroups, 96 / 112 / 128 per thread).  With TMA
// stores, eight 4 KB staging blocks sit beside the ring (4 stages for
// 192-256); 192 and 224 also come with 5 stages and direct stores, which
// long reductions prefer (the planner's choice, v.tma_out).  Every kernel
// takes the deepest ring that fits (tc_max_stages).
cudaError_t launch_tc_s32(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                          const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st) {
  const bool km = v.b_kmajor, t = v.tma_out != 0;
  switch (v.bn) {
    case 256: return km ? launch_one<256, tc_max_stages(256, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
                        : launch_one<256, tc_max_stages(256, 8, 1), false, kEpiS32, 8, 1>(a, b, o, w, p, grid, st);
    case 224:
      if (!km) return cudaErrorInvalidValue;
      return t ? launch_one<224, tc_max_stages(224, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
               : launch_one<224, tc_max_stages(224, 8, 0), true, kEpiS32, 8, 0>(a, b, o, w, p, grid, st);
    case 192:
      if (km)
        return t ? launch_one<192, tc_max_stages(192, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
                 : launch_one<192, tc_max_stages(192, 8, 0), true, kEpiS32, 8, 0>(a, b, o, w, p, grid, st);
      return t ? launch_one<192, tc_max_stages(192, 8, 1), false, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
               : launch_one<192, tc_max_stages(192, 8, 0), false, kEpiS32, 8, 0>(a, b, o, w, p, grid, st);
    case 128: return km ? launch_one<128, tc_max_stages(128, 4, 1), true, kEpiS32, 4, 1>(a, b, o, w, p, grid, st)
                        : launch_one<128, tc_max_stages(128, 4, 1), false, kEpiS32, 4, 1>(a, b, o, w, p, grid, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb300

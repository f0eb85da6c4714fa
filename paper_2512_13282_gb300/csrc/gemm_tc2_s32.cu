// Instantiations of the CTA-pair tcgen05 kernel with the exact int32 (slab)
// epilogue: TMA stores through eight 4 KB staging blocks (6 stages for
// 192-256, 8 for 128); 192 and 224 also come with direct stores and the
// deeper rings that frees (8 and 7 stages) for long reductions (the
// planner's choice, v.tma_out).  Every kernel takes the deepest ring that
// fits (tc_max_stages).
#include "gemm_tc2_launch.cuh"

namespace gb300 {

cudaError_t launch_tc2_s32(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st) {
  const bool t = v.tma_out != 0;
  if (v.b_kmajor) {
    switch (v.bn) {
      case 256: return launch_pair<256, tc_max_stages(256 / 2, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st);
      case 224: return t ? launch_pair<224, tc_max_stages(224 / 2, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
                         : launch_pair<224, tc_max_stages(224 / 2, 8, 0), true, kEpiS32, 8, 0>(a, b, o, w, p, grid, st);
      case 192: return t ? launch_pair<192, tc_max_stages(192 / 2, 8, 1), true, kEpiS32, 8, 1>(a, b, o, w, p, grid, st)
                         : launch_pair<192, tc_max_stages(192 / 2, 8, 0), true, kEpiS32, 8, 0>(a, b, o, w, p, grid, st);
      case 128: return launch_pair<128, tc_max_stages(128 / 2, 4, 1), true, kEpiS32, 4, 1>(a, b, o, w, p, grid, st);
    }
  } else {
    switch (v.bn) {
      case 256: return launch_pair<256, tc_max_stages(256 / 2, 8, 1), false, kEpiS32, 8, 1>(a, b, o, w, p, grid, st);
      case 128: return launch_pair<128, tc_max_stages(128 / 2, 4, 1), false, kEpiS32, 4, 1>(a, b, o, w, p, grid, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb300

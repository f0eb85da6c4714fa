// Instantiations of the CTA-pair tcgen05 kernel with the exact int32 (slab)
// epilogue.
#include "gemm_tc2_launch.cuh"

namespace gb300 {

cudaError_t launch_tc2_s32(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const TcParams &p, int grid, cudaStream_t st) {
  if (v.b_kmajor) {
    switch (v.bn) {
      case 256: return launch_pair<256, 6, true, kEpiS32, 8>(a, b, p, grid, st);
      case 224: return launch_pair<224, 7, true, kEpiS32, 8>(a, b, p, grid, st);
      case 192: return launch_pair<192, 7, true, kEpiS32, 8>(a, b, p, grid, st);
      case 128: return launch_pair<128, 8, true, kEpiS32, 4>(a, b, p, grid, st);
    }
  } else {
    switch (v.bn) {
      case 256: return launch_pair<256, 6, false, kEpiS32, 8>(a, b, p, grid, st);
      case 128: return launch_pair<128, 8, false, kEpiS32, 4>(a, b, p, grid, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb300

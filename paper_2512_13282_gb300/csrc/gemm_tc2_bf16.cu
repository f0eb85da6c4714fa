// Instantiations of the CTA-pair tcgen05 kernel with the bf16 epilogue.
#include "gemm_tc2_launch.cuh"

namespace gb300 {

// Pair tile widths (256 x BN per pair; BN/2 columns of B per CTA): 256 and
// 128 for either B layout, 224 and 192 for B column-major; TMA stores through
// 4 KB staging blocks, or 1 KB blocks for 224, which keeps its seventh stage.
// Every kernel takes the deepest ring that fits (tc_max_stages: 6, 7, 7, 8).
cudaError_t launch_tc2_bf16(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                            const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st) {
  if (v.b_kmajor) {
    switch (v.bn) {
      case 256: return launch_pair<256, tc_max_stages(256 / 2, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 224: return launch_pair<224, tc_max_stages(224 / 2, 4, 2), true, kEpiBf16, 4, 2>(a, b, o, w, p, grid, st);
      case 192: return launch_pair<192, tc_max_stages(192 / 2, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 128: return launch_pair<128, tc_max_stages(128 / 2, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
    }
  } else {
    switch (v.bn) {
      case 256: return launch_pair<256, tc_max_stages(256 / 2, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 128: return launch_pair<128, tc_max_stages(128 / 2, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
    }
  }
  return cudaErrorInvalidValue;
}

int tc2_bf16_tma_out(int bn) { return bn == 224 ? 2 : 1; }

int pair_slots() {
  // Co-resident SM pairs for a kernel holding one CTA per SM (all pair
  // variants use > 113 KB of shared memory), queried once per device.
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] > 0) return cached[dev];
  constexpr int kStages = tc_max_stages(256 / 2, 4, 1);
  using Cfg = Tc2Cfg<256, kStages, true, kEpiBf16, 4, 1>;
  auto kern = gemm_tc2_kernel<256, kStages, true, kEpiBf16, 4, 1>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(Cfg::kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) return 0;
  cached[dev] = n;
  return n;
}

}  // namespace gb300

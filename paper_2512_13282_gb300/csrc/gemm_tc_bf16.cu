// Instantiations of the tcgen05 kernel with the bf16 epilogue.
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

// Tile widths compiled for the bf16 epilogue, with their stage counts and
// output path (TMA stores through four 4 KB staging blocks, or, where those
// would cost a pipeline stage, through four 1 KB blocks of 16 columns):
// 64 (8, 4 KB), 96 (7, 4 KB; B column-major only), 128 (6, 4 KB), 192 (5,
// 4 KB), 224 (5, 1 KB; B column-major only), 256 (4, 4 KB) -- in each case
// the deepest ring that fits (tc_max_stages).  The narrow tiles serve
// memory-bound GEMMs with few rows: N / 96 tiles of 128 x 96 fill the SMs
// without a K split, and so without the reduction launch (bf16 128 x 11008
// x 4096: 115 CTAs), and 64 fits N = 64 without padding columns.
cudaError_t launch_tc_bf16(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st) {
  if (v.b_kmajor) {
    switch (v.bn) {
      case 256: return launch_one<256, tc_max_stages(256, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 224: return launch_one<224, tc_max_stages(224, 4, 2), true, kEpiBf16, 4, 2>(a, b, o, w, p, grid, st);
      case 192: return launch_one<192, tc_max_stages(192, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 128: return launch_one<128, tc_max_stages(128, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 96: return launch_one<96, tc_max_stages(96, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 64: return launch_one<64, tc_max_stages(64, 4, 1), true, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
    }
  } else {
    switch (v.bn) {
      case 256: return launch_one<256, tc_max_stages(256, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 192: return launch_one<192, tc_max_stages(192, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 128: return launch_one<128, tc_max_stages(128, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
      case 64: return launch_one<64, tc_max_stages(64, 4, 1), false, kEpiBf16, 4, 1>(a, b, o, w, p, grid, st);
    }
  }
  return cudaErrorInvalidValue;
}

// Output variant (1: 4 KB TMA staging blocks, 2: 1 KB) of launch_tc_bf16's
// kernel for this tile width.
int tc_bf16_tma_out(int bn) { return bn == 224 ? 2 : 1; }

}  // namespace gb300

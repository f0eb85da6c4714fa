// gemm_internal.h -- host-side declarations shared by the library's
// translation units (not part of the public ABI).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <utility>

#include "gb300_gemm.h"
#include "gemm_tc.cuh"

namespace gb300 {

// Whether kernels that consume the previous kernel's output (the tcgen05
// GEMM after operand staging, the split-K reduction after the GEMM) are
// launched with programmatic stream serialisation, so that their launch and
// set-up overlap the previous kernel's tail (GB300_GEMM_PDL=0 turns it off).
bool pdl_enabled();

// cudaLaunchKernelEx with programmatic stream serialisation when
// pdl_enabled(), plus a cluster dimension when cluster_x > 1.
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, int cluster_x,
                      Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = (unsigned)cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// One compiled variant of the tcgen05 kernel.
struct TcVariant {
  int bn;        // tile width (see the instantiation files for the compiled set)
  bool b_kmajor; // B stored N x K (K contiguous)
  int epi;       // kEpiBf16 or kEpiS32
  bool pair;     // CTA-pair kernel (256-row tiles, cta_group::2) or single CTA (128 rows)
  int tma_out;   // epilogue output variant: 0 direct stores, 1 TMA via 4 KB blocks, 2 TMA via 1 KB bf16 blocks
};

// Launch the persistent tcgen05 GEMM kernel (gemm_tc_bf16.cu / gemm_tc_s32.cu).
cudaError_t launch_tc_bf16(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st);
cudaError_t launch_tc_s32(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                          const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st);
// Output variant (TcVariant::tma_out) of the bf16 kernel of a tile width.
int tc_bf16_tma_out(int bn);
int tc2_bf16_tma_out(int bn);
// Number of CTA pairs that can be resident at once (0 if unknown).
int pair_slots();
// The CTA-pair kernel (gemm_tc2_bf16.cu / gemm_tc2_s32.cu); grid is even.
cudaError_t launch_tc2_bf16(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                            const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st);
cudaError_t launch_tc2_s32(const TcVariant &v, const CUtensorMap &a, const CUtensorMap &b,
                           const CUtensorMap &o, const CUtensorMap &w, const TcParams &p, int grid, cudaStream_t st);

// int8 GEMM for memory-bound shapes with the large operand converted to bf16
// inside the kernel (gemm_s8tm.cu).  P (int8, K contiguous, P_rows x K) is
// the operand streamed from HBM; Q (Q_rows x K) the small one, staged by
// launch_s8tm_stage_q as bf16 shared-memory images.  The sum over k of
// P[p][k] * Q[q][k] is C[q][p] when swap (P = B stored N x K, Q = A) and
// C[p][q] otherwise (P = A, Q = B).
constexpr int kS8tmKB = 128;  // K per k-block of gemm_s8tm_kernel
struct S8tmParams {
  int P_rows, Q_rows, K;
  int M, N;          // C extents
  int tiles_p, tiles_q;
  int num_kb;        // ceil(K / kS8tmKB)
  int splits, kb_per_split;
  int slab_kb;       // k-blocks per exact fp32 slab (1024 / kS8tmKB)
  int add_into_c;    // splits add their exact sums into C (int32, zeroed by the Q staging launch)
  int c_tma;         // ... with TMA reductions through tmC (else element by element)
  int swap;
  void *C;
  int64_t ldc;
  void *ws;          // split-K partials of int16 / int8 outputs: splits x M x N int32 (row pitch N);
                     // int32 outputs with split-K are added into C, zeroed beforehand
  uint32_t *err;
  uint64_t wait_limit_ns;
  int out_bits;      // 32, 16 or 8
  int out_shift;
  const void *q_img; // Q's images, tiles_q x num_kb of them (s8tm_q_image_bytes in all)
};
// Bytes of Q's images for QN = qn columns per tile.
size_t s8tm_q_image_bytes(int qn, int64_t Q_rows, int64_t K);
// Writes Q's images: Q(q, k) = src[q * sq + k * sk] (int8), exact bf16;
// when zero_c is not null, also sets the c_rows x c_cols int32 matrix at
// zero_c (row pitch ldc) to zero.
cudaError_t launch_s8tm_stage_q(const int8_t *src, int64_t sq, int64_t sk, int64_t Q_rows, int64_t K, int qn,
                                void *img, int32_t *zero_c, int64_t c_rows, int64_t c_cols, int64_t ldc,
                                cudaStream_t st);
// qn: 64 or 128 columns of Q per tile.  p_kmajor: P's rows are K
// contiguous (boxes of 128 k x 128 rows); otherwise P's rows are the
// contiguous dimension of its storage (boxes of 128 rows x 128 k, read
// transposed by the converters).
// tc maps int32 C (32 x 32 boxes, 128-byte swizzle) when p.c_tma is set.
cudaError_t launch_s8tm(int qn, bool p_kmajor, const CUtensorMap &tp, const CUtensorMap &tc, const S8tmParams &p,
                        int grid, cudaStream_t st);

// Auxiliary kernels (aux_kernels.cu).  Each returns the launch error.
// int8 -> bf16 (exact) of two matrices (A and B) in one launch; each is
// rows x cols with an arbitrary source leading dimension.
struct S8Job {
  const int8_t *src;
  int64_t rows, cols, ld_src;
  uint16_t *dst;
  int64_t ld_dst;
};
cudaError_t launch_s8_to_bf16_pair(const S8Job &a, const S8Job &b, int sms, cudaStream_t st);
// bf16 copy into an aligned buffer (re-pitching a misaligned operand).
cudaError_t launch_pack_u16(const uint16_t *src, int64_t rows, int64_t cols, int64_t ld_src,
                            uint16_t *dst, int64_t ld_dst, int sms, cudaStream_t st);
// Plain streaming read of `bytes` (16-byte aligned, a multiple of 16) with
// 16-byte loads over 4 blocks per SM; writes `sink` only in a case that does
// not occur for ordinary data (read-bandwidth diagnostic).
cudaError_t launch_read_stream(const void *p, size_t bytes, uint32_t *sink, int sms, cudaStream_t st);
// One-thread kernel whose bounded mbarrier wait is made to expire
// (failure-detection self-test).
cudaError_t launch_wait_timeout_probe(uint32_t *err, uint64_t limit_ns, cudaStream_t st);
// Fill an M x N block of 8-, 16- or 32-bit elements with zero.
cudaError_t launch_zero_fill(void *C, int64_t M, int64_t N, int64_t ldc, int esize, int sms,
                             cudaStream_t st);
// The part of C a split-K reduction covers: all of it (count == 0), or the
// `count` tiles of rows x cols (cols a multiple of 4) from raster position
// `first` on (raster_tile), the split tail of a tensor-core launch.
struct ReduceTiles {
  int first, count, tiles_m, tiles_n, group_m, rows, cols;
};
// Split-K reduction: C = round(sum over splits of ws[s]) (fp32 -> bf16 RNE)
// or C = sum of int32 partials, stored as int32 (out_bits 32) or
// requantised to out_bits = 16 / 8 with right shift `shift`; over the
// elements of C that rt covers.
cudaError_t launch_splitk_reduce_bf16(const float *ws, int splits, int64_t M, int64_t N,
                                      uint16_t *C, int64_t ldc, const ReduceTiles &rt, cudaStream_t st);
cudaError_t launch_splitk_reduce_s32(const int32_t *ws, int splits, int64_t M, int64_t N, void *C,
                                     int64_t ldc, int out_bits, int shift, const ReduceTiles &rt,
                                     cudaStream_t st);

// Argument checks of the int8 entry points (no CUDA calls).
gemm_status_t validate_s8(int64_t M, int64_t N, int64_t K, const void *A, int64_t lda, const void *B,
                          int64_t ldb, int b_layout, const void *C, int64_t ldc);

// Forgets the no-allocation scratch address cached for device `dev`
// (gemm_noalloc.cu).
void noalloc_forget_device(int dev);

// The int8 GEMM with its staging and split-K scratch in caller-provided
// device memory of `capacity` bytes (gemm_api.cu; used by gemm_noalloc.cu).
gemm_status_t s8_gemm_into_scratch(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                                   const int8_t *B, int64_t ldb, int b_layout, int32_t *C, int64_t ldc,
                                   cudaStream_t st, void *scratch, size_t capacity);

// Exact int8 GEMM of a small problem in one launch on the CUDA cores
// (gemm_tiny.cu): 32 x 32 tiles of C, __dp4a over K.
struct TinyParams {
  const int8_t *A;
  int64_t lda;
  const int8_t *B;
  int64_t ldb;
  void *C;
  int64_t ldc;
  int64_t M, N, K;
  int out_bits;   // 32 (int32 C), 16 or 8 (requantised C)
  int out_shift;  // right shift of requantised outputs, 0..31
};
cudaError_t launch_tiny_s8(const TinyParams &p, bool row_b, cudaStream_t st);

// Small-M GEMM on the CUDA cores (gemm_skinny.cu).  M <= 16.
struct SkinnyParams {
  const void *A;
  int64_t lda;
  const void *B;
  int64_t ldb;
  void *C;
  int64_t ldc;
  int M;
  int64_t N, K;
  int kb;              // rows of K per block slice (skinny_geometry)
  int ks;              // slices (blocks per column strip)
  int b_align;         // 16, 8, 4, 2 or 1: alignment in bytes of the B base and row pitch
  void *ws;            // ks x M x N 32-bit partials (ks > 1)
  uint32_t *tickets;   // one zeroed counter per column strip (ks > 1)
  int out_bits;        // int8: 32 (int32 C), 16 or 8 (requantised C)
  int out_shift;       // int8 with out_bits < 32: right shift, 0..31
};
// Column strips of the launch (the grid's x); fills kb and ks.
int64_t skinny_geometry(int M, int64_t N, int64_t K, bool int8, bool row_b, int sms, int *kb, int *ks);
cudaError_t launch_skinny(const SkinnyParams &p, bool int8, bool row_b, int64_t strips, cudaStream_t st);

}  // namespace gb300

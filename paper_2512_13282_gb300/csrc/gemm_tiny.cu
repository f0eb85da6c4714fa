// gemm_tiny.cu -- exact int8 GEMM for problems too small to fill the GPU, in
// one launch on the CUDA cores.
//
// Below a few hundred million multiply-adds the time of an int8 GEMM is the
// launch and the memory latency, not the arithmetic: the tensor-core path
// needs two launches (the operands are staged as bf16 first) and a pipeline
// start per tile, while `__dp4a` (four exact int8 products summed into an
// exact int32 per instruction) reads the int8 operands as they are.  Each
// block computes a 32 x 32 tile of C with 256 threads (2 x 2 outputs each),
// stepping through K in slabs of 512: every load of a slab (A's 32 rows, B's
// 32 columns) is issued before the first one is used, so a slab costs one
// memory latency, and the slab is placed in shared memory as 32-bit words of
// four consecutive k, a row-major B being byte-transposed on the way (four
// k-rows x four columns per thread).
// Every partial sum of at most 131071 products fits int32, so the result is
// exact; it is stored as int32 or requantised to int16 / int8 like the other
// int8 paths.
#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kTT = 32;         // tile rows and columns
constexpr int kTK = 512;        // K per slab: every load of a slab is issued before any is used
constexpr int kTThreads = 256;
constexpr int kTW = kTK / 4;    // words of four k per row of a slab
constexpr int kTPad = kTW + 1;  // padded row: conflict-free column reads

// Four int8 of row `r`, k0 .. k0 + 3 of a row-major operand (row pitch ld),
// zero outside [0, rows) x [0, cols); one 32-bit load when aligned.
__device__ __forceinline__ uint32_t load4_row(const int8_t *p, int64_t ld, int64_t rows, int64_t cols, int64_t r,
                                              int64_t k0) {
  if (r >= rows || k0 >= cols) return 0u;
  const int8_t *q = p + r * ld + k0;
  if (k0 + 4 <= cols && (reinterpret_cast<uintptr_t>(q) & 3) == 0) return __ldg(reinterpret_cast<const uint32_t *>(q));
  uint32_t w = 0;
  for (int i = 0; i < 4; ++i)
    if (k0 + i < cols) w |= (uint32_t)(uint8_t)q[i] << (8 * i);
  return w;
}

// Sixteen int8 (four words) of row `r` from k0: one 16-byte load when the
// piece lies inside the row and is aligned, else word by word.
__device__ __forceinline__ uint4 load16_row(const int8_t *p, int64_t ld, int64_t rows, int64_t cols, int64_t r,
                                            int64_t k0) {
  if (r < rows && k0 + 16 <= cols) {
    const int8_t *q = p + r * ld + k0;
    if ((reinterpret_cast<uintptr_t>(q) & 15) == 0) return __ldg(reinterpret_cast<const uint4 *>(q));
  }
  return make_uint4(load4_row(p, ld, rows, cols, r, k0), load4_row(p, ld, rows, cols, r, k0 + 4),
                    load4_row(p, ld, rows, cols, r, k0 + 8), load4_row(p, ld, rows, cols, r, k0 + 12));
}

template <bool ROW_B>
__global__ void __launch_bounds__(kTThreads) gemm_tiny_s8_kernel(const TinyParams p) {
  __shared__ uint32_t As[kTT][kTPad];
  __shared__ uint32_t Bs[kTT][kTPad];
  // launched with programmatic dependent launch: the next kernel of the
  // stream may be scheduled now; global memory is touched only once the
  // previous kernel has completed
  griddep_launch_dependents();
  griddep_wait();
  const int tid = threadIdx.x;
  const int ty = tid >> 4, tx = tid & 15;
  const int64_t m0 = (int64_t)blockIdx.y * kTT, n0 = (int64_t)blockIdx.x * kTT;
  int32_t acc[2][2] = {{0, 0}, {0, 0}};
  for (int64_t k0 = 0; k0 < p.K; k0 += kTK) {
    // A: 32 rows x 32 pieces of 16 bytes, four per thread, all in flight
    // before any is stored
    uint4 a[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = tid + i * kTThreads, r = e >> 5, piece = e & 31;
      a[i] = load16_row(p.A, p.lda, p.M, p.K, m0 + r, k0 + 16 * piece);
    }
    uint4 b[4];
    if constexpr (!ROW_B) {
      // B stored N x K: the same as A, rows are columns of C
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = tid + i * kTThreads, c = e >> 5, piece = e & 31;
        b[i] = load16_row(p.B, p.ldb, p.N, p.K, n0 + c, k0 + 16 * piece);
      }
    } else {
      // B stored K x N: four blocks of 4 k-rows x 4 columns per thread (of
      // 128 x 8 in the slab), one word per k-row
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = tid + i * kTThreads, cq = e & 7, kq = e >> 3;
        const int64_t k = k0 + 4 * kq;
        b[i] = make_uint4(load4_row(p.B, p.ldb, p.K, p.N, k, n0 + 4 * cq),
                          load4_row(p.B, p.ldb, p.K, p.N, k + 1, n0 + 4 * cq),
                          load4_row(p.B, p.ldb, p.K, p.N, k + 2, n0 + 4 * cq),
                          load4_row(p.B, p.ldb, p.K, p.N, k + 3, n0 + 4 * cq));
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = tid + i * kTThreads, r = e >> 5, w = 4 * (e & 31);
      As[r][w] = a[i].x;
      As[r][w + 1] = a[i].y;
      As[r][w + 2] = a[i].z;
      As[r][w + 3] = a[i].w;
    }
    if constexpr (!ROW_B) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = tid + i * kTThreads, c = e >> 5, w = 4 * (e & 31);
        Bs[c][w] = b[i].x;
        Bs[c][w + 1] = b[i].y;
        Bs[c][w + 2] = b[i].z;
        Bs[c][w + 3] = b[i].w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int e = tid + i * kTThreads, cq = e & 7, kq = e >> 3;
        // byte j of word t is B(k + t, n0 + 4 cq + j); column j's word takes
        // byte j of the four words, k ascending from the low byte
        const uint32_t lo01 = __byte_perm(b[i].x, b[i].y, 0x5140), hi01 = __byte_perm(b[i].x, b[i].y, 0x7362);
        const uint32_t lo23 = __byte_perm(b[i].z, b[i].w, 0x5140), hi23 = __byte_perm(b[i].z, b[i].w, 0x7362);
        Bs[4 * cq + 0][kq] = __byte_perm(lo01, lo23, 0x5410);
        Bs[4 * cq + 1][kq] = __byte_perm(lo01, lo23, 0x7632);
        Bs[4 * cq + 2][kq] = __byte_perm(hi01, hi23, 0x5410);
        Bs[4 * cq + 3][kq] = __byte_perm(hi01, hi23, 0x7632);
      }
    }
    __syncthreads();
    const int wn = (int)min((int64_t)kTW, (p.K - k0 + 3) / 4);  // words of this slab holding k < K
#pragma unroll 8
    for (int w = 0; w < wn; ++w) {
      const int a0 = (int)As[ty][w], a1 = (int)As[ty + 16][w];
      const int b0 = (int)Bs[tx][w], b1 = (int)Bs[tx + 16][w];
      acc[0][0] = __dp4a(a0, b0, acc[0][0]);
      acc[0][1] = __dp4a(a0, b1, acc[0][1]);
      acc[1][0] = __dp4a(a1, b0, acc[1][0]);
      acc[1][1] = __dp4a(a1, b1, acc[1][1]);
    }
    __syncthreads();
  }
  const int32_t hi = p.out_bits == 32 ? 0 : (1 << (p.out_bits - 1)) - 1, lo = -hi - 1;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int64_t m = m0 + ty + 16 * i;
    if (m >= p.M) continue;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int64_t n = n0 + tx + 16 * j;
      if (n >= p.N) continue;
      const int64_t at = m * p.ldc + n;
      if (p.out_bits == 32)
        static_cast<int32_t *>(p.C)[at] = acc[i][j];
      else if (p.out_bits == 16)
        static_cast<int16_t *>(p.C)[at] = (int16_t)requantize_s32(acc[i][j], p.out_shift, lo, hi);
      else
        static_cast<int8_t *>(p.C)[at] = (int8_t)requantize_s32(acc[i][j], p.out_shift, lo, hi);
    }
  }
}

}  // namespace

cudaError_t launch_tiny_s8(const TinyParams &p, bool row_b, cudaStream_t st) {
  const dim3 grid((unsigned)((p.N + kTT - 1) / kTT), (unsigned)((p.M + kTT - 1) / kTT));
  return row_b ? launch_ex(gemm_tiny_s8_kernel<true>, grid, dim3(kTThreads), 0, st, 1, p)
               : launch_ex(gemm_tiny_s8_kernel<false>, grid, dim3(kTThreads), 0, st, 1, p);
}

}  // namespace gb300

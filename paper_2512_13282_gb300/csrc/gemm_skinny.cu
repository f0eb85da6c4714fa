// gemm_skinny.cu -- C = A.B for very small M (M <= 16) on the CUDA cores.
//
// With a handful of rows in A the product is a few matrix-vector products:
// every element of B is used M times, far too few for the tensor cores to
// matter, and the time is the time to stream B from HBM once (the paper
// lists GEMV as future work, Sec. 5.3.4).  This kernel streams B with
// coalesced loads, many in flight per lane, and keeps A in shared memory:
//
//   - B row-major (K x N): a lane owns 4, 8 or 16 contiguous bytes of columns
//     and walks rows k; a warp reads 128-512 contiguous bytes per row.  The
//     lane width, the bytes a lane has in flight and the blocks per SM
//     depend on M and the type (rowb_shape), and the grid is one wave.
//   - B column-major (N x K): a warp owns 4 columns (rows of the storage)
//     and its lanes split K in 16-byte chunks; partial dot products are
//     summed across lanes at the end.
//   - int8 uses __dp4a (4 exact int8 products summed into int32); a row-major
//     B piece of 4 rows x 4 columns is byte-transposed so that each word holds
//     4 consecutive k of one column.  bf16 accumulates in fp32 FMAs.
//   - K is split across the 8 warps of a block and across `ks` blocks per
//     column strip; the last block of a strip to finish (atomic ticket) adds
//     the fp32/int32 partials of all blocks in a fixed order, so results do
//     not depend on scheduling, and rounds once to bf16.
#include <cuda_bf16.h>

#include <type_traits>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kSkThreads = 256;
constexpr int kSkWarps = kSkThreads / 32;

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// 32-bit partial word of output (m, n) of block slice `slice`.
__device__ __forceinline__ uint32_t *partial_ptr(const SkinnyParams &p, int slice, int m, int64_t n) {
  return reinterpret_cast<uint32_t *>(p.ws) + ((int64_t)slice * p.M + m) * p.N + n;
}

// The block's contribution for output columns [n0, n0 + cols): written as
// the final result when ks == 1, else as partials with a last-block sum.
// `vals` is this block's (already warp-combined) M x cols result in shared
// memory, row stride `ld` words.
// One int8-path result: int32, or requantised to int16 / int8.
__device__ __forceinline__ void store_s8_out(const SkinnyParams &p, int m, int64_t n, int32_t s) {
  const int64_t at = m * p.ldc + n;
  if (p.out_bits == 32) {
    reinterpret_cast<int32_t *>(p.C)[at] = s;
  } else {
    const int32_t hi = (1 << (p.out_bits - 1)) - 1, lo = -hi - 1;
    const int32_t q = requantize_s32(s, p.out_shift, lo, hi);
    if (p.out_bits == 16)
      reinterpret_cast<int16_t *>(p.C)[at] = (int16_t)q;
    else
      reinterpret_cast<int8_t *>(p.C)[at] = (int8_t)q;
  }
}

template <bool INT8>
__device__ void finish_block(const SkinnyParams &p, const uint32_t *vals, int ld, int64_t n0, int cols,
                             uint32_t *ticket_smem) {
  const int total = p.M * cols;
  if (p.ks == 1) {
    for (int t = threadIdx.x; t < total; t += kSkThreads) {
      const int m = t / cols, c = t - m * cols;
      const int64_t n = n0 + c;
      if (INT8) {
        store_s8_out(p, m, n, (int32_t)vals[m * ld + c]);
      } else {
        __nv_bfloat16 h = __float2bfloat16_rn(__uint_as_float(vals[m * ld + c]));
        reinterpret_cast<uint16_t *>(p.C)[m * p.ldc + n] = *reinterpret_cast<uint16_t *>(&h);
      }
    }
    return;
  }
  const int slice = blockIdx.y;
  for (int t = threadIdx.x; t < total; t += kSkThreads) {
    const int m = t / cols, c = t - m * cols;
    *partial_ptr(p, slice, m, n0 + c) = vals[m * ld + c];
  }
  __threadfence();  // partials visible device-wide before the ticket
  __syncthreads();
  if (threadIdx.x == 0) *ticket_smem = atomicAdd(&p.tickets[blockIdx.x], 1u);
  __syncthreads();
  if (*ticket_smem != (uint32_t)(p.ks - 1)) return;
  // last block of this strip: sum all slices in order 0..ks-1
  __threadfence();
  for (int t = threadIdx.x; t < total; t += kSkThreads) {
    const int m = t / cols, c = t - m * cols;
    const int64_t n = n0 + c;
    // slices 0, 1, ... in order, four loads in flight at a time
    uint32_t v[4];
    int k = 0;
    if (INT8) {
      int32_t s = 0;
      for (; k + 4 <= p.ks; k += 4) {
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __ldcg(partial_ptr(p, k + i, m, n));
#pragma unroll
        for (int i = 0; i < 4; ++i) s += (int32_t)v[i];
      }
      for (; k < p.ks; ++k) s += (int32_t)__ldcg(partial_ptr(p, k, m, n));
      store_s8_out(p, m, n, s);
    } else {
      float s = 0.f;
      for (; k + 4 <= p.ks; k += 4) {
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __ldcg(partial_ptr(p, k + i, m, n));
#pragma unroll
        for (int i = 0; i < 4; ++i) s += __uint_as_float(v[i]);
      }
      for (; k < p.ks; ++k) s += __uint_as_float(__ldcg(partial_ptr(p, k, m, n)));
      __nv_bfloat16 h = __float2bfloat16_rn(s);
      reinterpret_cast<uint16_t *>(p.C)[m * p.ldc + n] = *reinterpret_cast<uint16_t *>(&h);
    }
  }
  if (threadIdx.x == 0) p.tickets[blockIdx.x] = 0u;  // ready for the next call
}

// ------------------------------------------------------------ B row-major
// A lane owns VB contiguous bytes of every row it reads (VB / esize columns)
// and a warp 32 * VB bytes: the block's column strip.  The block's K slice is
// cut into batches of R = RB / VB rows; warp w takes batches w, w + 8, ...
// Each batch is loaded in two halves, and a half is reloaded with the next
// batch's rows as soon as it has been multiplied, so every lane keeps RB / 2
// to RB bytes of B in flight.  The first loads are issued before A is staged
// in shared memory.  int8 byte-transposes each 4-row x 4-column piece so that
// a word holds four k of one column for __dp4a.
constexpr int mt_of(int M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16; }

// Launch shape of the row-major kernel per rows of A held (MT) and type:
// bytes of a B row a lane loads (VB), bytes a lane loads per batch (RB) and
// resident blocks per SM (BPS, which caps the registers a thread at 64, 80
// or 128).  Chosen on GB300 by timing every (VB, RB, BPS) on M = 1, 4, 8, 16
// with N = 4096..11008, K = 4096: narrower lanes with more blocks win for
// int8 (8-byte lanes, 16 KB of B in flight per block, 4 blocks per SM at
// M = 1; 4-byte lanes, 8 KB per block, at M = 8), wider lanes for bf16,
// whose fp32 accumulators leave fewer registers.
struct RowBShape {
  int vb, rb, bps;
};
constexpr RowBShape rowb_shape(int mt, bool int8) {
  return int8 ? (mt == 1 ? RowBShape{8, 128, 4} : mt == 2 ? RowBShape{8, 128, 3} : mt == 4 ? RowBShape{8, 128, 2}
                 : RowBShape{4, 64, mt == 8 ? 3 : 2})
              : (mt == 1 ? RowBShape{8, 128, 4} : mt == 2 ? RowBShape{8, 128, 3} : mt <= 8 ? RowBShape{8, 128, 2}
                 : RowBShape{4, 128, 2});
}

template <int MT, int VB, bool INT8, int RB, int BPS>
__global__ void __launch_bounds__(kSkThreads, BPS) skinny_rowB_kernel(const SkinnyParams p) {
  constexpr int R = RB / VB;              // rows per batch
  constexpr int H = R / 2;                // rows per half batch (a multiple of 4)
  static_assert(H >= 1 && (!INT8 || H % 4 == 0), "int8 half batches are whole quads of rows");
  constexpr int W = VB / 4;               // 32-bit words per lane per row
  constexpr int CPL = INT8 ? VB : VB / 2; // columns per lane
  constexpr int kCols = 32 * CPL;         // columns per block
  constexpr int esize = INT8 ? 1 : 2;
  extern __shared__ uint32_t sk_smem[];
  __shared__ uint32_t ticket;
  // launched with programmatic dependent launch: the next kernel of the
  // stream may be scheduled now, and this one touches global memory only
  // once the previous one has completed
  griddep_launch_dependents();
  griddep_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n0 = (int64_t)blockIdx.x * kCols;
  const int64_t k0 = (int64_t)blockIdx.y * p.kb;
  const int kb = (int)min((int64_t)p.kb, p.K - k0);  // rows of this slice (> 0)
  const int batches = (kb + R - 1) / R;
  const int64_t col = n0 + lane * CPL;
  const bool vec = p.b_align >= VB && col + CPL <= p.N;
  const uint8_t *Bb = reinterpret_cast<const uint8_t *>(p.B) + (k0 * p.ldb + col) * esize;
  const int64_t pitch = p.ldb * esize;

  // rows [r0, r0 + H) of the slice into w (zero past the slice and past N)
  auto load_half = [&](int r0, uint32_t (&w)[H][W]) {
#pragma unroll
    for (int r = 0; r < H; ++r) {
#pragma unroll
      for (int j = 0; j < W; ++j) w[r][j] = 0u;
      if (r0 + r >= kb) continue;
      const uint8_t *row = Bb + (int64_t)(r0 + r) * pitch;
      if (vec) {
        if constexpr (VB == 16) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row));
          w[r][0] = v.x; w[r][1] = v.y; w[r][2] = v.z; w[r][3] = v.w;
        } else if constexpr (VB == 8) {
          const uint2 v = __ldcs(reinterpret_cast<const uint2 *>(row));
          w[r][0] = v.x; w[r][1] = v.y;
        } else {
          w[r][0] = __ldcs(reinterpret_cast<const unsigned int *>(row));
        }
      } else {
#pragma unroll
        for (int c = 0; c < CPL; ++c)
          if (col + c < p.N) {
            const uint32_t v = INT8 ? (uint32_t)row[c] : (uint32_t)reinterpret_cast<const uint16_t *>(row)[c];
            w[(r)][(c * esize) >> 2] |= v << (8 * ((c * esize) & 3));
          }
      }
    }
  };

  uint32_t h0[H][W], h1[H][W];
  int b = warp;
  load_half(b * R, h0);
  load_half(b * R + H, h1);

  // stage A[0:M, k0:k0+kb] (zero for m >= M and past the slice, up to whole
  // batches): int8 as words of 4 k, bf16 as fp32
  const int kbp = batches * R;
  const int words = kbp / 4;
  uint32_t *a_s = sk_smem;
  if constexpr (INT8) {
    for (int t = threadIdx.x; t < MT * words; t += kSkThreads) {
      const int m = t / words, q = t - m * words;
      uint32_t v = 0;
      if (m < p.M) {
        const int8_t *a = reinterpret_cast<const int8_t *>(p.A) + (int64_t)m * p.lda + k0 + 4 * q;
        for (int i = 0; i < 4; ++i)
          if (4 * q + i < kb) v |= (uint32_t)(uint8_t)a[i] << (8 * i);
      }
      a_s[t] = v;
    }
  } else {
    for (int t = threadIdx.x; t < MT * kbp; t += kSkThreads) {
      const int m = t / kbp, k = t - m * kbp;
      float v = 0.f;
      if (m < p.M && k < kb)
        v = __uint_as_float((uint32_t)reinterpret_cast<const uint16_t *>(p.A)[(int64_t)m * p.lda + k0 + k] << 16);
      a_s[t] = __float_as_uint(v);
    }
  }
  __syncthreads();

  using Acc = typename std::conditional<INT8, int32_t, float>::type;
  Acc acc[MT][CPL];
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int c = 0; c < CPL; ++c) acc[m][c] = 0;

  // multiply rows [r0, r0 + H) held in w
  auto mul_half = [&](int r0, const uint32_t (&w)[H][W]) {
    if constexpr (INT8) {
#pragma unroll
      for (int q = 0; q < H / 4; ++q) {
        const int aq = (r0 >> 2) + q;  // A word of these four rows
#pragma unroll
        for (int j = 0; j < W; ++j) {
          const uint32_t x0 = w[4 * q][j], x1 = w[4 * q + 1][j], x2 = w[4 * q + 2][j], x3 = w[4 * q + 3][j];
          const uint32_t lo01 = __byte_perm(x0, x1, 0x5140), hi01 = __byte_perm(x0, x1, 0x7362);
          const uint32_t lo23 = __byte_perm(x2, x3, 0x5140), hi23 = __byte_perm(x2, x3, 0x7362);
          const uint32_t cw[4] = {__byte_perm(lo01, lo23, 0x5410), __byte_perm(lo01, lo23, 0x7632),
                                  __byte_perm(hi01, hi23, 0x5410), __byte_perm(hi01, hi23, 0x7632)};
#pragma unroll
          for (int m = 0; m < MT; ++m) {
            const int aw = (int)a_s[m * words + aq];
#pragma unroll
            for (int c = 0; c < 4; ++c)
              acc[m][4 * j + c] = __dp4a(aw, (int)cw[c], acc[m][4 * j + c]);
          }
        }
      }
    } else {
#pragma unroll
      for (int r = 0; r < H; ++r) {
        float bv[CPL];
#pragma unroll
        for (int j = 0; j < W; ++j) {
          bv[2 * j] = bf16_lo(w[r][j]);
          bv[2 * j + 1] = bf16_hi(w[r][j]);
        }
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          const float a = __uint_as_float(a_s[m * kbp + r0 + r]);
#pragma unroll
          for (int c = 0; c < CPL; ++c) acc[m][c] = fmaf(a, bv[c], acc[m][c]);
        }
      }
    }
  };

  for (; b < batches; b += kSkWarps) {
    const int nb = b + kSkWarps;
    if (b * R < kb) mul_half(b * R, h0);
    if (nb < batches) load_half(nb * R, h0);
    if (b * R + H < kb) mul_half(b * R + H, h1);
    if (nb < batches) load_half(nb * R + H, h1);
  }

  // combine the 8 warps: int8 by shared-memory atomics (integer sums do not
  // depend on order), bf16 through one slot per warp summed in warp order
  __syncthreads();  // every warp is done with the A slice
  uint32_t *red = sk_smem;
  const int cols = (int)min((int64_t)kCols, p.N - n0);
  if constexpr (INT8) {
    for (int t = threadIdx.x; t < MT * kCols; t += kSkThreads) red[t] = 0u;
    __syncthreads();
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int c = 0; c < CPL; ++c) atomicAdd(reinterpret_cast<int *>(&red[m * kCols + lane * CPL + c]), (int)acc[m][c]);
    __syncthreads();
    finish_block<true>(p, red, kCols, n0, cols, &ticket);
  } else {
    float *slot = reinterpret_cast<float *>(sk_smem) + MT * kCols * warp;
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int c = 0; c < CPL; ++c) slot[m * kCols + lane * CPL + c] = (float)acc[m][c];
    __syncthreads();
    float *sum = reinterpret_cast<float *>(sk_smem) + MT * kCols * kSkWarps;
    for (int t = threadIdx.x; t < MT * kCols; t += kSkThreads) {
      float s = 0.f;
#pragma unroll
      for (int w2 = 0; w2 < kSkWarps; ++w2) s += reinterpret_cast<const float *>(sk_smem)[MT * kCols * w2 + t];
      sum[t] = s;
    }
    __syncthreads();
    finish_block<false>(p, reinterpret_cast<uint32_t *>(sum), kCols, n0, cols, &ticket);
  }
}

// --------------------------------------------------------- B column-major
// Block = 32 columns (4 per warp) x a K range; lanes split the range in
// 16-byte chunks of the B rows (the storage rows are the columns of B).
// Resident blocks per SM of the column-major kernel, 5 down to 2 as its
// registers grow with M (48 to 128 a thread).
constexpr int colb_blocks(int mt) { return mt == 1 ? 5 : mt <= 4 ? 4 : mt == 8 ? 3 : 2; }

template <int MT, bool INT8>
__global__ void __launch_bounds__(kSkThreads, colb_blocks(MT)) skinny_colB_kernel(const SkinnyParams p) {
  constexpr int kColsPerWarp = 4;
  constexpr int kCols = kColsPerWarp * kSkWarps;  // 32
  constexpr int kElems = INT8 ? 16 : 8;            // elements per 16-byte chunk
  extern __shared__ uint32_t sk_smem[];
  __shared__ uint32_t ticket;
  griddep_launch_dependents();  // programmatic dependent launch, as above
  griddep_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n0 = (int64_t)blockIdx.x * kCols;
  const int64_t k0 = (int64_t)blockIdx.y * p.kb;
  const int kb = (int)min((int64_t)p.kb, (int64_t)p.K - k0);
  const int chunks = (kb + kElems - 1) / kElems;
  // A slice in shared memory as 16-byte chunks: MT x chunks x 4 words
  uint32_t *a_s = sk_smem;
  for (int t = threadIdx.x; t < MT * chunks * 4; t += kSkThreads) {
    const int m = t / (chunks * 4), r = t - m * chunks * 4;
    uint32_t v = 0;
    if (m < p.M) {
      if (INT8) {
        const int8_t *a = reinterpret_cast<const int8_t *>(p.A) + (int64_t)m * p.lda + k0;
        for (int i = 0; i < 4; ++i)
          if (4 * r + i < kb) v |= (uint32_t)(uint8_t)a[4 * r + i] << (8 * i);
      } else {
        const uint16_t *a = reinterpret_cast<const uint16_t *>(p.A) + (int64_t)m * p.lda + k0;
        for (int i = 0; i < 2; ++i)
          if (2 * r + i < kb) v |= (uint32_t)a[2 * r + i] << (16 * i);
      }
    }
    a_s[t] = v;
  }
  __syncthreads();

  uint32_t acc[MT][kColsPerWarp];  // int32 or fp32 bits
  float facc[MT][kColsPerWarp];
  int32_t iacc[MT][kColsPerWarp];
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int j = 0; j < kColsPerWarp; ++j) {
      facc[m][j] = 0.f;
      iacc[m][j] = 0;
    }
  for (int ch = lane; ch < chunks; ch += 32) {
    const int kk = ch * kElems;
    uint32_t w[kColsPerWarp][4];
#pragma unroll
    for (int j = 0; j < kColsPerWarp; ++j) {
      w[j][0] = w[j][1] = w[j][2] = w[j][3] = 0;
      const int64_t n = n0 + warp * kColsPerWarp + j;
      if (n >= p.N) continue;
      if (INT8) {
        const int8_t *row = reinterpret_cast<const int8_t *>(p.B) + n * p.ldb + k0 + kk;
        if (p.b_align >= 16 && kk + kElems <= kb) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row));
          w[j][0] = v.x; w[j][1] = v.y; w[j][2] = v.z; w[j][3] = v.w;
        } else {
          for (int i = 0; i < kElems; ++i)
            if (kk + i < kb) w[j][i >> 2] |= (uint32_t)(uint8_t)row[i] << (8 * (i & 3));
        }
      } else {
        const uint16_t *row = reinterpret_cast<const uint16_t *>(p.B) + n * p.ldb + k0 + kk;
        if (p.b_align >= 16 && kk + kElems <= kb) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row));
          w[j][0] = v.x; w[j][1] = v.y; w[j][2] = v.z; w[j][3] = v.w;
        } else {
          for (int i = 0; i < kElems; ++i)
            if (kk + i < kb) w[j][i >> 1] |= (uint32_t)row[i] << (16 * (i & 1));
        }
      }
    }
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const uint4 av = *reinterpret_cast<const uint4 *>(&a_s[(m * chunks + ch) * 4]);
      const uint32_t a[4] = {av.x, av.y, av.z, av.w};
#pragma unroll
      for (int j = 0; j < kColsPerWarp; ++j)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (INT8) {
            iacc[m][j] = __dp4a((int)a[i], (int)w[j][i], iacc[m][j]);
          } else {
            facc[m][j] = fmaf(bf16_lo(a[i]), bf16_lo(w[j][i]), facc[m][j]);
            facc[m][j] = fmaf(bf16_hi(a[i]), bf16_hi(w[j][i]), facc[m][j]);
          }
        }
    }
  }
  // sum across lanes (fixed butterfly order)
#pragma unroll
  for (int m = 0; m < MT; ++m)
#pragma unroll
    for (int j = 0; j < kColsPerWarp; ++j) {
      if (INT8) {
        int32_t v = iacc[m][j];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        acc[m][j] = (uint32_t)v;
      } else {
        float v = facc[m][j];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        acc[m][j] = __float_as_uint(v);
      }
    }
  __syncthreads();
  uint32_t *red = sk_smem;  // MT x 32
  if (lane == 0)
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int j = 0; j < kColsPerWarp; ++j) red[m * kCols + warp * kColsPerWarp + j] = acc[m][j];
  __syncthreads();
  const int cols = (int)min((int64_t)kCols, (int64_t)p.N - n0);
  finish_block<INT8>(p, red, kCols, n0, cols, &ticket);
}

template <int MT, bool INT8>
cudaError_t launch_mt(const SkinnyParams &p, dim3 grid, bool row_b, cudaStream_t st) {
  if (row_b) {
    constexpr RowBShape sh = rowb_shape(MT, INT8);
    constexpr int VB = sh.vb;
    constexpr int kCols = 32 * (INT8 ? VB : VB / 2);
    const size_t a_bytes = INT8 ? (size_t)MT * p.kb : (size_t)MT * p.kb * 4;  // kb: whole batches
    const size_t red_bytes = (size_t)MT * kCols * 4 * (INT8 ? 1 : kSkWarps + 1);
    const size_t smem = a_bytes > red_bytes ? a_bytes : red_bytes;
    auto kern = skinny_rowB_kernel<MT, VB, INT8, sh.rb, sh.bps>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_ex(kern, grid, dim3(kSkThreads), smem, st, 1, p);
    if (e != cudaSuccess) return e;
  } else {
    const int kelems = INT8 ? 16 : 8;
    const size_t a_bytes = (size_t)MT * ((p.kb + kelems - 1) / kelems) * 16;
    const size_t red_bytes = (size_t)MT * 32 * 4;
    const size_t smem = a_bytes > red_bytes ? a_bytes : red_bytes;
    auto kern = skinny_colB_kernel<MT, INT8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_ex(kern, grid, dim3(kSkThreads), smem, st, 1, p);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace

// Column strips, rows of K per block slice and slices.
//  - Row-major B: one wave of blocks, as many slices as the resident blocks
//    (rowb_shape) leave room for beside the column strips; slices are whole
//    multiples of the block's 8 batches and hold at most 32 KB of A.
//  - Column-major B: about four blocks per SM, slices a multiple of 32 rows,
//    at most 2048.
// Either way the fp32/int32 partial sums a slice writes (4 bytes per
// output) stay below 1/8 of the B bytes it reads (kb >= 32 * M / esize).
int64_t skinny_geometry(int M, int64_t N, int64_t K, bool int8, bool row_b, int sms, int *kb, int *ks) {
  const int mt = mt_of(M), esize = int8 ? 1 : 2;
  const RowBShape sh = rowb_shape(mt, int8);
  const int64_t cols = row_b ? 32 * (sh.vb / esize) : 32;
  const int64_t strips = (N + cols - 1) / cols;
  const int64_t unit = row_b ? 8 * (sh.rb / sh.vb) : 32;
  const int64_t max_rows = row_b ? (32768 / (mt * (int8 ? 1 : 4))) / unit * unit : 2048;
  const int64_t min_rows = ((32 * (int64_t)(row_b ? mt : M) + esize - 1) / esize + unit - 1) / unit * unit;
  int64_t s = row_b ? (int64_t)sms * sh.bps / strips                  // one wave
                    : ((int64_t)sms * 4 + strips - 1) / strips;
  const int64_t max_s = (K + min_rows - 1) / min_rows;
  if (s > max_s) s = max_s;
  if (s < 1) s = 1;
  int64_t rows = (K + s - 1) / s;
  rows = (rows + unit - 1) / unit * unit;
  if (rows > max_rows) rows = max_rows;
  *kb = (int)rows;
  *ks = (int)((K + rows - 1) / rows);
  return strips;
}

cudaError_t launch_skinny(const SkinnyParams &p, bool int8, bool row_b, int64_t strips, cudaStream_t st) {
  const dim3 grid((unsigned)strips, (unsigned)p.ks, 1);
  switch (mt_of(p.M)) {
    case 1: return int8 ? launch_mt<1, true>(p, grid, row_b, st) : launch_mt<1, false>(p, grid, row_b, st);
    case 2: return int8 ? launch_mt<2, true>(p, grid, row_b, st) : launch_mt<2, false>(p, grid, row_b, st);
    case 4: return int8 ? launch_mt<4, true>(p, grid, row_b, st) : launch_mt<4, false>(p, grid, row_b, st);
    case 8: return int8 ? launch_mt<8, true>(p, grid, row_b, st) : launch_mt<8, false>(p, grid, row_b, st);
    default: return int8 ? launch_mt<16, true>(p, grid, row_b, st) : launch_mt<16, false>(p, grid, row_b, st);
  }
}

}  // namespace gb300

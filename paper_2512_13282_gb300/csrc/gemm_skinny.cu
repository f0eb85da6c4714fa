// gemm_skinny.cu -- C = A.B for very small M (M <= 16) on the CUDA cores.
//
// With a handful of rows in A the product is a few matrix-vector products:
// every element of B is used M times, far too few for the tensor cores to
// matter, and the time is the time to stream B from HBM once (the paper
// lists GEMV as future work, Sec. 5.3.4).  This kernel streams B with
// 16-byte coalesced loads and keeps A in shared memory:
//
//   - B row-major (K x N): a lane owns 8 consecutive columns and walks rows
//     k; a warp reads 256 contiguous bf16 (or 32 lanes x 8 int8) per row.
//   - B column-major (N x K): a warp owns 4 columns (rows of the storage)
//     and its lanes split K in 16-byte chunks; partial dot products are
//     summed across lanes at the end.
//   - int8 uses __dp4a (4 exact int8 products summed into int32); a row-major
//     B chunk of 4 rows x 8 columns is byte-transposed so that each word holds
//     4 consecutive k of one column.  bf16 accumulates in fp32 FMAs.
//   - K is split across the 8 warps of a block and across `ks` blocks per
//     column strip; the last block of a strip to finish (atomic ticket) adds
//     the fp32/int32 partials of all blocks in a fixed order, so results do
//     not depend on scheduling, and rounds once to bf16.
#include <cuda_bf16.h>

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
    if (INT8) {
      int32_t s = 0;
      for (int k = 0; k < p.ks; ++k) s += (int32_t)__ldcg(partial_ptr(p, k, m, n));
      store_s8_out(p, m, n, s);
    } else {
      float s = 0.f;
      for (int k = 0; k < p.ks; ++k) s += __uint_as_float(__ldcg(partial_ptr(p, k, m, n)));
      __nv_bfloat16 h = __float2bfloat16_rn(s);
      reinterpret_cast<uint16_t *>(p.C)[m * p.ldc + n] = *reinterpret_cast<uint16_t *>(&h);
    }
  }
  if (threadIdx.x == 0) p.tickets[blockIdx.x] = 0u;  // ready for the next call
}

// ------------------------------------------------------------ B row-major
// Block = 256 columns (8 per lane) x a K range; warp w takes rows
// k0 + w, k0 + w + 8, ... of the range.  MT = rows of A held (>= M).
template <int MT, bool INT8>
__global__ void __launch_bounds__(kSkThreads) skinny_rowB_kernel(const SkinnyParams p) {
  constexpr int kCols = 256;
  extern __shared__ uint32_t sk_smem[];
  uint32_t *a_s = sk_smem;                        // A slice: MT x kb (bf16 as fp32 bits, or int8 words)
  __shared__ uint32_t ticket;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n0 = (int64_t)blockIdx.x * kCols;
  const int64_t k0 = (int64_t)blockIdx.y * p.kb;
  const int kb = (int)min((int64_t)p.kb, (int64_t)p.K - k0);  // rows of this slice (> 0)
  // stage A[0:M, k0:k0+kb] (zero for m >= M)
  if (INT8) {
    const int words = (kb + 3) / 4;
    for (int t = threadIdx.x; t < MT * words; t += kSkThreads) {
      const int m = t / words, w = t - m * words;
      uint32_t v = 0;
      if (m < p.M) {
        const int8_t *a = reinterpret_cast<const int8_t *>(p.A) + (int64_t)m * p.lda + k0 + 4 * w;
        for (int i = 0; i < 4; ++i)
          if (4 * w + i < kb) v |= (uint32_t)(uint8_t)a[i] << (8 * i);
      }
      a_s[m * words + w] = v;
    }
  } else {
    for (int t = threadIdx.x; t < MT * kb; t += kSkThreads) {
      const int m = t / kb, k = t - m * kb;
      float v = 0.f;
      if (m < p.M) v = __uint_as_float((uint32_t)reinterpret_cast<const uint16_t *>(p.A)[(int64_t)m * p.lda + k0 + k] << 16);
      a_s[m * kb + k] = __float_as_uint(v);
    }
  }
  __syncthreads();

  const int64_t col = n0 + lane * 8;
  const bool vec = col + 8 <= p.N && p.b_vec;
  if (INT8) {
    int32_t acc[MT][8];
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[m][c] = 0;
    const int8_t *B = reinterpret_cast<const int8_t *>(p.B);
    const int words = (kb + 3) / 4;
    // warp w handles k-quads 2w, 2w+1, then +16, ...: 8 rows in flight
    for (int qbase = 2 * warp; qbase < words; qbase += 2 * kSkWarps) {
      uint32_t lo[2][4], hi[2][4];  // 8 columns of 4 rows, two quads
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          lo[h][i] = hi[h][i] = 0;
          const int kq = 4 * (qbase + h) + i;
          if (kq >= kb) continue;
          const int8_t *row = B + (k0 + kq) * p.ldb + col;
          if (vec) {
            const uint2 v = __ldcs(reinterpret_cast<const uint2 *>(row));
            lo[h][i] = v.x;
            hi[h][i] = v.y;
          } else {
            for (int c = 0; c < 8; ++c)
              if (col + c < p.N) {
                const uint32_t b = (uint8_t)row[c];
                if (c < 4) lo[h][i] |= b << (8 * c); else hi[h][i] |= b << (8 * (c - 4));
              }
          }
        }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int q = qbase + h;
        if (q >= words) break;
        // byte transpose: column word c = bytes c of rows 0..3
        uint32_t cw[8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          // bytes [x.c, y.c] of two rows, then [r0.c, r1.c, r2.c, r3.c]
          const uint32_t sel = (uint32_t)c | ((uint32_t)(c + 4) << 4);
          const uint32_t s01 = __byte_perm(lo[h][0], lo[h][1], sel);
          const uint32_t s23 = __byte_perm(lo[h][2], lo[h][3], sel);
          cw[c] = __byte_perm(s01, s23, 0x5410);
          const uint32_t t01 = __byte_perm(hi[h][0], hi[h][1], sel);
          const uint32_t t23 = __byte_perm(hi[h][2], hi[h][3], sel);
          cw[4 + c] = __byte_perm(t01, t23, 0x5410);
        }
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          const int aw = (int)a_s[m * words + q];
#pragma unroll
          for (int c = 0; c < 8; ++c) acc[m][c] = __dp4a(aw, (int)cw[c], acc[m][c]);
        }
      }
    }
    // combine the 8 warps in shared memory (reuse the A area after a sync)
    __syncthreads();
    uint32_t *red = sk_smem;  // MT x 256 words
    for (int t = threadIdx.x; t < MT * kCols; t += kSkThreads) red[t] = 0u;
    __syncthreads();
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int c = 0; c < 8; ++c) atomicAdd(reinterpret_cast<int *>(&red[m * kCols + lane * 8 + c]), acc[m][c]);
    __syncthreads();
    const int cols = (int)min((int64_t)kCols, (int64_t)p.N - n0);
    finish_block<true>(p, red, kCols, n0, cols, &ticket);
  } else {
    float acc[MT][8];
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[m][c] = 0.f;
    const uint16_t *B = reinterpret_cast<const uint16_t *>(p.B);
    constexpr int kRows = 4;  // rows in flight per lane
    for (int kbase = warp * kRows; kbase < kb; kbase += kSkWarps * kRows) {
      uint32_t w[kRows][4];
#pragma unroll
      for (int r = 0; r < kRows; ++r) {
        w[r][0] = w[r][1] = w[r][2] = w[r][3] = 0;
        const int k = kbase + r;
        if (k >= kb) continue;
        const uint16_t *row = B + (k0 + k) * p.ldb + col;
        if (vec) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row));
          w[r][0] = v.x; w[r][1] = v.y; w[r][2] = v.z; w[r][3] = v.w;
        } else {
          for (int c = 0; c < 8; ++c)
            if (col + c < p.N) w[r][c >> 1] |= (uint32_t)row[c] << (16 * (c & 1));
        }
      }
#pragma unroll
      for (int r = 0; r < kRows; ++r) {
        const int k = kbase + r;
        if (k >= kb) break;
        float b[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          b[2 * i] = bf16_lo(w[r][i]);
          b[2 * i + 1] = bf16_hi(w[r][i]);
        }
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          const float a = __uint_as_float(a_s[m * kb + k]);
#pragma unroll
          for (int c = 0; c < 8; ++c) acc[m][c] = fmaf(a, b[c], acc[m][c]);
        }
      }
    }
    // combine the 8 warps in a fixed order (warp 0, 1, ...) in shared memory
    __syncthreads();
    float *red = reinterpret_cast<float *>(sk_smem);  // MT x 256
    for (int w2 = 0; w2 < kSkWarps; ++w2) {
      if (warp == w2) {
#pragma unroll
        for (int m = 0; m < MT; ++m)
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            float &r = red[m * kCols + lane * 8 + c];
            r = (w2 == 0) ? acc[m][c] : r + acc[m][c];
          }
      }
      __syncthreads();
    }
    const int cols = (int)min((int64_t)kCols, (int64_t)p.N - n0);
    finish_block<false>(p, reinterpret_cast<uint32_t *>(red), kCols, n0, cols, &ticket);
  }
}

// --------------------------------------------------------- B column-major
// Block = 32 columns (4 per warp) x a K range; lanes split the range in
// 16-byte chunks of the B rows (the storage rows are the columns of B).
template <int MT, bool INT8>
__global__ void __launch_bounds__(kSkThreads) skinny_colB_kernel(const SkinnyParams p) {
  constexpr int kColsPerWarp = 4;
  constexpr int kCols = kColsPerWarp * kSkWarps;  // 32
  constexpr int kElems = INT8 ? 16 : 8;            // elements per 16-byte chunk
  extern __shared__ uint32_t sk_smem[];
  __shared__ uint32_t ticket;
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
        if (p.b_vec && kk + kElems <= kb) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row));
          w[j][0] = v.x; w[j][1] = v.y; w[j][2] = v.z; w[j][3] = v.w;
        } else {
          for (int i = 0; i < kElems; ++i)
            if (kk + i < kb) w[j][i >> 2] |= (uint32_t)(uint8_t)row[i] << (8 * (i & 3));
        }
      } else {
        const uint16_t *row = reinterpret_cast<const uint16_t *>(p.B) + n * p.ldb + k0 + kk;
        if (p.b_vec && kk + kElems <= kb) {
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
    const size_t a_bytes = INT8 ? (size_t)MT * ((p.kb + 3) / 4) * 4 : (size_t)MT * p.kb * 4;
    const size_t red_bytes = (size_t)MT * 256 * 4;
    const size_t smem = a_bytes > red_bytes ? a_bytes : red_bytes;
    auto kern = skinny_rowB_kernel<MT, INT8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kSkThreads, smem, st>>>(p);
  } else {
    const int kelems = INT8 ? 16 : 8;
    const size_t a_bytes = (size_t)MT * ((p.kb + kelems - 1) / kelems) * 16;
    const size_t red_bytes = (size_t)MT * 32 * 4;
    const size_t smem = a_bytes > red_bytes ? a_bytes : red_bytes;
    auto kern = skinny_colB_kernel<MT, INT8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kSkThreads, smem, st>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace

// Rows of K per block slice, and slices, for `strips` column strips: enough
// blocks to cover the SMs a few times over, while the fp32/int32 partial
// sums a slice writes (4 bytes per output) stay below 1/8 of the B bytes it
// reads (kb >= 32 * m_rows / esize); slices are a multiple of 32 rows.
void skinny_split(int64_t K, int64_t strips, int sms, int m_rows, int esize, int *kb, int *ks) {
  const int64_t want_blocks = (int64_t)sms * 4;
  int64_t s = (want_blocks + strips - 1) / strips;
  const int64_t min_rows = (32 * (int64_t)m_rows + esize - 1) / esize;
  const int64_t max_s = (K + (min_rows > 32 ? min_rows : 32) - 1) / (min_rows > 32 ? min_rows : 32);
  if (s > max_s) s = max_s;
  if (s < 1) s = 1;
  int64_t rows = (K + s - 1) / s;
  rows = (rows + 31) / 32 * 32;
  if (rows > 2048) rows = 2048;  // bounds the A slice in shared memory
  *kb = (int)rows;
  *ks = (int)((K + rows - 1) / rows);
}

cudaError_t launch_skinny(const SkinnyParams &p, bool int8, bool row_b, cudaStream_t st) {
  const int64_t cols_per_block = row_b ? 256 : 32;
  const dim3 grid((unsigned)((p.N + cols_per_block - 1) / cols_per_block), (unsigned)p.ks, 1);
  const int mt = p.M <= 1 ? 1 : p.M <= 2 ? 2 : p.M <= 4 ? 4 : p.M <= 8 ? 8 : 16;
  switch (mt) {
    case 1: return int8 ? launch_mt<1, true>(p, grid, row_b, st) : launch_mt<1, false>(p, grid, row_b, st);
    case 2: return int8 ? launch_mt<2, true>(p, grid, row_b, st) : launch_mt<2, false>(p, grid, row_b, st);
    case 4: return int8 ? launch_mt<4, true>(p, grid, row_b, st) : launch_mt<4, false>(p, grid, row_b, st);
    case 8: return int8 ? launch_mt<8, true>(p, grid, row_b, st) : launch_mt<8, false>(p, grid, row_b, st);
    default: return int8 ? launch_mt<16, true>(p, grid, row_b, st) : launch_mt<16, false>(p, grid, row_b, st);
  }
}

}  // namespace gb300

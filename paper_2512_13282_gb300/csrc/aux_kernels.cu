// aux_kernels.cu -- the memory-bound helpers around the tensor-core kernel:
// operand staging (int8 -> bf16, re-pitching misaligned bf16), zero fill for
// K == 0, and the split-K reduction.
#include <cuda_bf16.h>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kThreads = 256;

inline int grid_for(int64_t work, int per_thread, int sms) {
  const int64_t want = (work + (int64_t)kThreads * per_thread - 1) / ((int64_t)kThreads * per_thread);
  const int64_t cap = (int64_t)sms * 8;
  return (int)(want < 1 ? 1 : (want > cap ? cap : want));
}

// int8 -> bf16 bit pattern.  |v| <= 128 needs 8 significant bits, which a
// bf16 has, so the float's upper half is the exact bf16 (low half is zero).
__device__ __forceinline__ uint32_t s8_to_bf16_bits(int v) {
  return __float_as_uint(static_cast<float>(v)) >> 16;
}

// Each thread converts 16 consecutive elements of a row.
__global__ void s8_to_bf16_kernel(const int8_t *__restrict__ src, int64_t rows, int64_t cols,
                                  int64_t ld_src, uint16_t *__restrict__ dst, int64_t ld_dst) {
  const int64_t chunks_per_row = (cols + 15) / 16;
  const int64_t total = rows * chunks_per_row;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = t / chunks_per_row;
    const int64_t c = (t - r * chunks_per_row) * 16;
    const int8_t *s = src + r * ld_src + c;
    uint16_t *d = dst + r * ld_dst + c;
    if (c + 16 <= cols && (reinterpret_cast<uintptr_t>(s) & 15) == 0 &&
        (reinterpret_cast<uintptr_t>(d) & 15) == 0) {
      const int4 raw = __ldg(reinterpret_cast<const int4 *>(s));
      const uint32_t w[4] = {(uint32_t)raw.x, (uint32_t)raw.y, (uint32_t)raw.z, (uint32_t)raw.w};
      uint32_t o[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int b0 = (int8_t)(w[i] & 0xFF), b1 = (int8_t)((w[i] >> 8) & 0xFF);
        const int b2 = (int8_t)((w[i] >> 16) & 0xFF), b3 = (int8_t)(w[i] >> 24);
        o[2 * i] = s8_to_bf16_bits(b0) | (s8_to_bf16_bits(b1) << 16);
        o[2 * i + 1] = s8_to_bf16_bits(b2) | (s8_to_bf16_bits(b3) << 16);
      }
      uint4 *dv = reinterpret_cast<uint4 *>(d);
      dv[0] = make_uint4(o[0], o[1], o[2], o[3]);
      dv[1] = make_uint4(o[4], o[5], o[6], o[7]);
    } else {
      const int64_t n = cols - c < 16 ? cols - c : 16;
      for (int64_t i = 0; i < n; ++i) d[i] = (uint16_t)s8_to_bf16_bits(s[i]);
    }
  }
}

__global__ void pack_u16_kernel(const uint16_t *__restrict__ src, int64_t rows, int64_t cols,
                                int64_t ld_src, uint16_t *__restrict__ dst, int64_t ld_dst) {
  const int64_t total = rows * cols;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = t / cols, c = t - r * cols;
    dst[r * ld_dst + c] = src[r * ld_src + c];
  }
}

template <typename T>
__global__ void zero_fill_kernel(T *C, int64_t M, int64_t N, int64_t ldc) {
  const int64_t total = M * N;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = t / N, c = t - r * N;
    C[r * ldc + c] = T(0);
  }
}

// Sum the fp32 partials of all splits (fixed order: split 0, 1, ...), then
// round once to bf16, nearest even.
__global__ void splitk_reduce_bf16_kernel(const float *__restrict__ ws, int splits, int64_t M,
                                          int64_t N, uint16_t *__restrict__ C, int64_t ldc) {
  const int64_t total = M * N;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += ws[(int64_t)k * total + t];
    const int64_t r = t / N, c = t - r * N;
    __nv_bfloat16 h = __float2bfloat16_rn(s);
    C[r * ldc + c] = *reinterpret_cast<uint16_t *>(&h);
  }
}

__global__ void splitk_reduce_s32_kernel(const int32_t *__restrict__ ws, int splits, int64_t M,
                                         int64_t N, int32_t *__restrict__ C, int64_t ldc) {
  const int64_t total = M * N;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int32_t s = 0;
    for (int k = 0; k < splits; ++k) s += ws[(int64_t)k * total + t];
    const int64_t r = t / N, c = t - r * N;
    C[r * ldc + c] = s;
  }
}

}  // namespace

cudaError_t launch_s8_to_bf16(const int8_t *src, int64_t rows, int64_t cols, int64_t ld_src,
                              uint16_t *dst, int64_t ld_dst, int sms, cudaStream_t st) {
  const int64_t work = rows * ((cols + 15) / 16);
  s8_to_bf16_kernel<<<grid_for(work, 1, sms), kThreads, 0, st>>>(src, rows, cols, ld_src, dst, ld_dst);
  return cudaGetLastError();
}

cudaError_t launch_pack_u16(const uint16_t *src, int64_t rows, int64_t cols, int64_t ld_src,
                            uint16_t *dst, int64_t ld_dst, int sms, cudaStream_t st) {
  pack_u16_kernel<<<grid_for(rows * cols, 4, sms), kThreads, 0, st>>>(src, rows, cols, ld_src, dst, ld_dst);
  return cudaGetLastError();
}

cudaError_t launch_zero_fill(void *C, int64_t M, int64_t N, int64_t ldc, int esize, int sms,
                             cudaStream_t st) {
  const int g = grid_for(M * N, 4, sms);
  if (esize == 2)
    zero_fill_kernel<uint16_t><<<g, kThreads, 0, st>>>(static_cast<uint16_t *>(C), M, N, ldc);
  else
    zero_fill_kernel<int32_t><<<g, kThreads, 0, st>>>(static_cast<int32_t *>(C), M, N, ldc);
  return cudaGetLastError();
}

cudaError_t launch_splitk_reduce_bf16(const float *ws, int splits, int64_t M, int64_t N,
                                      uint16_t *C, int64_t ldc, int sms, cudaStream_t st) {
  splitk_reduce_bf16_kernel<<<grid_for(M * N, 2, sms), kThreads, 0, st>>>(ws, splits, M, N, C, ldc);
  return cudaGetLastError();
}

cudaError_t launch_splitk_reduce_s32(const int32_t *ws, int splits, int64_t M, int64_t N,
                                     int32_t *C, int64_t ldc, int sms, cudaStream_t st) {
  splitk_reduce_s32_kernel<<<grid_for(M * N, 2, sms), kThreads, 0, st>>>(ws, splits, M, N, C, ldc);
  return cudaGetLastError();
}

}  // namespace gb300

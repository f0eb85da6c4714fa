// aux_kernels.cu -- the memory-bound helpers around the tensor-core kernel:
// operand staging (int8 -> bf16, re-pitching misaligned bf16), zero fill for
// K == 0, and the split-K reduction (with the int8 path's requantisation).
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

// Converts 16 int8 held in a uint4 to 16 bf16 bit patterns in two uint4.
__device__ __forceinline__ void s8x16_to_bf16x16(const int4 raw, uint4 &lo, uint4 &hi) {
  const uint32_t w[4] = {(uint32_t)raw.x, (uint32_t)raw.y, (uint32_t)raw.z, (uint32_t)raw.w};
  uint32_t o[8];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int b0 = (int8_t)(w[i] & 0xFF), b1 = (int8_t)((w[i] >> 8) & 0xFF);
    const int b2 = (int8_t)((w[i] >> 16) & 0xFF), b3 = (int8_t)(w[i] >> 24);
    o[2 * i] = s8_to_bf16_bits(b0) | (s8_to_bf16_bits(b1) << 16);
    o[2 * i + 1] = s8_to_bf16_bits(b2) | (s8_to_bf16_bits(b3) << 16);
  }
  lo = make_uint4(o[0], o[1], o[2], o[3]);
  hi = make_uint4(o[4], o[5], o[6], o[7]);
}

constexpr int kS8Chunk = 32;       // int8 elements per work item
constexpr int kS8Threads = 256;

// Both matrices as one flat list of work items: item t < items_a is chunk
// t % cpr_a of row t / cpr_a of A (cpr = chunks per row, 32 elements each),
// the rest likewise of B.  A grid-stride loop over one resident wave of
// blocks covers wide and narrow matrices alike.  Aligned full chunks use two
// 16-byte loads and four 16-byte stores.  The next kernel (the GEMM) may be
// scheduled at once: it waits for this grid's completion before reading.
__global__ void __launch_bounds__(kS8Threads)
    s8_to_bf16_pair_kernel(const S8Job a, const S8Job b, int64_t cpr_a, int64_t cpr_b, int64_t items_a,
                           int64_t items) {
  griddep_launch_dependents();
  for (int64_t t = (int64_t)blockIdx.x * kS8Threads + threadIdx.x; t < items;
       t += (int64_t)gridDim.x * kS8Threads) {
    const bool in_a = t < items_a;
    const int64_t u = in_a ? t : t - items_a;
    const int64_t cpr = in_a ? cpr_a : cpr_b;
    const int64_t r = u / cpr;
    const int64_t c = (u - r * cpr) * kS8Chunk;
    const int64_t cols = in_a ? a.cols : b.cols;
    const int8_t *src = (in_a ? a.src : b.src) + r * (in_a ? a.ld_src : b.ld_src) + c;
    uint16_t *dst = (in_a ? a.dst : b.dst) + r * (in_a ? a.ld_dst : b.ld_dst) + c;
    const bool full = c + kS8Chunk <= cols;
    if (full && (reinterpret_cast<uintptr_t>(src) & 15) == 0 && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
      const int4 r0 = __ldg(reinterpret_cast<const int4 *>(src));
      const int4 r1 = __ldg(reinterpret_cast<const int4 *>(src) + 1);
      uint4 o0, o1, o2, o3;
      s8x16_to_bf16x16(r0, o0, o1);
      s8x16_to_bf16x16(r1, o2, o3);
      uint4 *dv = reinterpret_cast<uint4 *>(dst);
      dv[0] = o0;
      dv[1] = o1;
      dv[2] = o2;
      dv[3] = o3;
    } else {
      const int64_t n = cols - c < kS8Chunk ? cols - c : kS8Chunk;
      for (int64_t i = 0; i < n; ++i) dst[i] = (uint16_t)s8_to_bf16_bits(src[i]);
    }
  }
}

// Dense fast path: both matrices contiguous (leading dimension = columns,
// source 16-byte aligned), so each is one flat array; thread v converts
// 16-element vector v (v < va: of A, else of B) with one 16-byte load and
// two 16-byte stores, over a grid that covers every vector once (measured on
// GB300 faster than fewer threads looping over several vectors).  A last
// partial vector (elements % 16) is converted element by element.
__global__ void __launch_bounds__(kS8Threads)
    s8_to_bf16_dense_kernel(const S8Job a, const S8Job b, int64_t na, int64_t nb) {
  griddep_launch_dependents();
  const int64_t va = (na + 15) / 16, vtot = va + (nb + 15) / 16;
  const int64_t v = (int64_t)blockIdx.x * kS8Threads + threadIdx.x;
  if (v >= vtot) return;
  const bool in_a = v < va;
  const S8Job &j = in_a ? a : b;
  const int64_t n = in_a ? na : nb;
  const int64_t e = (in_a ? v : v - va) * 16;
  if (e + 16 <= n) {
    const int4 raw = __ldcs(reinterpret_cast<const int4 *>(j.src + e));
    uint4 lo, hi;
    s8x16_to_bf16x16(raw, lo, hi);
    uint4 *d = reinterpret_cast<uint4 *>(j.dst + e);
    d[0] = lo;
    d[1] = hi;
  } else {
    for (int64_t i = e; i < n; ++i) j.dst[i] = (uint16_t)s8_to_bf16_bits(j.src[i]);
  }
}

__global__ void pack_u16_kernel(const uint16_t *__restrict__ src, int64_t rows, int64_t cols,
                                int64_t ld_src, uint16_t *__restrict__ dst, int64_t ld_dst) {
  griddep_launch_dependents();  // the GEMM waits for completion before reading
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
  griddep_wait();  // the partials come from the GEMM launched just before
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

// Sum the int32 partials; store as int32, or requantised to int16 / int8.
__global__ void splitk_reduce_s32_kernel(const int32_t *__restrict__ ws, int splits, int64_t M,
                                         int64_t N, void *__restrict__ C, int64_t ldc, int out_bits,
                                         int shift) {
  griddep_wait();
  const int64_t total = M * N;
  const int32_t hi = out_bits == 32 ? INT32_MAX : (1 << (out_bits - 1)) - 1, lo = -hi - 1;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    int32_t s = 0;
    for (int k = 0; k < splits; ++k) s += ws[(int64_t)k * total + t];
    const int64_t r = t / N, c = t - r * N;
    if (out_bits == 32)
      static_cast<int32_t *>(C)[r * ldc + c] = s;
    else if (out_bits == 16)
      static_cast<int16_t *>(C)[r * ldc + c] = (int16_t)requantize_s32(s, shift, lo, hi);
    else
      static_cast<int8_t *>(C)[r * ldc + c] = (int8_t)requantize_s32(s, shift, lo, hi);
  }
}

// One thread waits, with the GEMM kernels' bounded wait, on an mbarrier that
// nothing will ever arrive on: the wait gives up after limit_ns and records
// the timeout in the device error word, exactly as a stalled GEMM would.
__global__ void wait_timeout_probe_kernel(uint32_t *err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_addr(&bar), 1);
    abort_flag = 0u;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) (void)mbar_wait(smem_addr(&bar), 0, &abort_flag, err, limit_ns);
}

}  // namespace

cudaError_t launch_wait_timeout_probe(uint32_t *err, uint64_t limit_ns, cudaStream_t st) {
  wait_timeout_probe_kernel<<<1, 32, 0, st>>>(err, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_s8_to_bf16_pair(const S8Job &a, const S8Job &b, int sms, cudaStream_t st) {
  static int blocks_per_sm = 0;  // resident blocks per SM (same on every GB300)
  if (blocks_per_sm == 0) {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, s8_to_bf16_pair_kernel, kS8Threads, 0) != cudaSuccess ||
        n < 1)
      n = 4;
    blocks_per_sm = n;
  }
  auto dense = [](const S8Job &j) {
    return j.ld_src == j.cols && j.ld_dst == j.cols && (reinterpret_cast<uintptr_t>(j.src) & 15) == 0 &&
           (reinterpret_cast<uintptr_t>(j.dst) & 15) == 0;
  };
  if (dense(a) && dense(b)) {
    const int64_t na = a.rows * a.cols, nb = b.rows * b.cols;
    const int64_t vecs = (na + 15) / 16 + (nb + 15) / 16;
    if (vecs == 0) return cudaSuccess;
    s8_to_bf16_dense_kernel<<<(unsigned)((vecs + kS8Threads - 1) / kS8Threads), kS8Threads, 0, st>>>(a, b, na, nb);
    return cudaGetLastError();
  }
  const int64_t cpr_a = (a.cols + kS8Chunk - 1) / kS8Chunk, cpr_b = (b.cols + kS8Chunk - 1) / kS8Chunk;
  const int64_t items_a = a.rows * cpr_a, items = items_a + b.rows * cpr_b;
  if (items == 0) return cudaSuccess;
  const int64_t want = (items + kS8Threads - 1) / kS8Threads;
  const int64_t wave = (int64_t)sms * blocks_per_sm;
  const unsigned grid = (unsigned)(want < wave ? want : wave);
  s8_to_bf16_pair_kernel<<<grid, kS8Threads, 0, st>>>(a, b, cpr_a, cpr_b, items_a, items);
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
  if (esize == 1)
    zero_fill_kernel<uint8_t><<<g, kThreads, 0, st>>>(static_cast<uint8_t *>(C), M, N, ldc);
  else if (esize == 2)
    zero_fill_kernel<uint16_t><<<g, kThreads, 0, st>>>(static_cast<uint16_t *>(C), M, N, ldc);
  else
    zero_fill_kernel<int32_t><<<g, kThreads, 0, st>>>(static_cast<int32_t *>(C), M, N, ldc);
  return cudaGetLastError();
}

cudaError_t launch_splitk_reduce_bf16(const float *ws, int splits, int64_t M, int64_t N,
                                      uint16_t *C, int64_t ldc, int sms, cudaStream_t st) {
  return launch_ex(splitk_reduce_bf16_kernel, dim3(grid_for(M * N, 2, sms)), dim3(kThreads), 0, st, 1, ws, splits,
                   M, N, C, ldc);
}

cudaError_t launch_splitk_reduce_s32(const int32_t *ws, int splits, int64_t M, int64_t N, void *C,
                                     int64_t ldc, int out_bits, int shift, int sms, cudaStream_t st) {
  return launch_ex(splitk_reduce_s32_kernel, dim3(grid_for(M * N, 2, sms)), dim3(kThreads), 0, st, 1, ws, splits,
                   M, N, C, ldc, out_bits, shift);
}

}  // namespace gb300

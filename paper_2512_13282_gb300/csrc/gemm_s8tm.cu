// gemm_s8tm.cu -- exact int8 GEMM for memory-bound shapes: one operand is
// converted to bf16 inside the kernel, straight into tensor memory.
//
// When one operand is much larger than the other (a few rows of
// activations against a weight matrix, or a weight matrix a few columns
// wide), the time is the time to stream the large operand from HBM once.
// The general int8 path first stages both operands as bf16 (one launch that
// reads 1 byte and writes 2 per element), then the GEMM reads those 2 bytes
// again: 5 bytes of traffic per element of the large operand instead of 1.
// This kernel stages only the small operand and streams the large one as
// int8:
//
//   P  the large operand, int8, K contiguous: B stored N x K when M is
//      small (P row = column n of C), or A when N is small (P row = row m).
//      It is the MMA's 128-row A operand, read from TMEM.
//   Q  the small operand, staged as bf16 beforehand (K-major or MN-major);
//      the MMA's QN-column B operand, read from shared memory.
//
// Roles (10 warps):
//   warp 0 (one lane)  TMA producer: per k-block of 128 a 128 x 128 int8
//                      box of P (128-byte rows, 128-byte swizzle) and two
//                      QN x 64 bf16 boxes of Q into a STAGES-deep
//                      shared-memory ring.  A P row of the box is one
//                      128-byte request: the number of row requests an SM
//                      can have served, not their bytes, bounds how fast it
//                      streams from HBM (measured on GB300: 64-byte rows
//                      gave half the bytes per second of 128-byte rows).
//   warps 6..9         converters: lane r of the warp with TMEM lane
//                      quadrant q converts P row 32 q + r (128 int8, read
//                      with eight conflict-free 16-byte loads) to 64 packed
//                      bf16 pairs and writes them to one of NA P slots in
//                      TMEM (tcgen05.st, lane = row, the lower k of a pair
//                      in the low half).
//   warp 1 (one lane)  MMA issuer: tcgen05.mma kind::f16 with A in TMEM and
//                      B in shared memory, into one of two TMEM accumulators
//                      of QN fp32 columns.
//   warps 2..5         epilogue: lane r of quadrant q owns P row 32 q + r.
//
// Exactness is the general int8 path's: every product is at most 2^14 in
// magnitude, so a partial sum of at most 1024 of them is an integer below
// 2^24 in magnitude and exact in fp32; the MMA warp closes the accumulator
// every 8 k-blocks of 128 (1024 K elements) and the epilogue converts each slab to
// int32 (exactly) and adds the slabs in int32 registers.
//
// A stage of the ring is free again once the MMAs that read its Q box have
// completed (tcgen05.commit) and every converter warp has read its P box
// (one arrival per warp): the empty barrier counts 1 + 4 arrivals.
#include <cuda_bf16.h>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kConvWarps = 4;
constexpr int kEpiWarps = 4;
constexpr int kThreadsS8tm = (2 + kEpiWarps + kConvWarps) * 32;  // 320
constexpr int kKB = kS8tmKB;                                      // K per k-block (stage)
constexpr uint32_t kPBytes = kBM * kKB;                           // 128 rows x 128 int8

template <int QN, bool Q_KMAJOR, int STAGES, int NA>
struct S8tmCfg {
  static_assert(QN == 64 || QN == 128, "QN is 64 or 128");
  static constexpr uint32_t kQHalf = QN * kRowBytes;  // QN x 64 bf16: one box of Q
  static constexpr uint32_t kQBytes = 2 * kQHalf;      // the k-block's two halves
  static constexpr uint32_t kStageBytes = kPBytes + kQBytes;
  static constexpr uint32_t kPOffset = 0;
  static constexpr uint32_t kQOffset = STAGES * kPBytes;  // 1024-byte aligned
  static constexpr uint32_t kBarOffset = kQOffset + STAGES * kQBytes;
  static constexpr uint32_t kNumBars = 2 * STAGES + 2 * NA + 5;
  static constexpr uint32_t kSmemBytes = kBarOffset + kNumBars * 8 + 16 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA is 227 KB");
  static constexpr uint32_t kPCol0 = 2 * QN;  // P slots (64 columns each) follow the two accumulators
  static constexpr uint32_t kTmemCols = pow2_at_least(2 * QN + 64 * NA);
  static_assert(kTmemCols <= 512, "TMEM has 512 columns");
};

struct S8tmUnit {
  int tp, tq, split, kb0, kb1;
};

__device__ __forceinline__ S8tmUnit decode_s8tm(const S8tmParams &p, int u) {
  const int tiles = p.tiles_p * p.tiles_q;
  S8tmUnit w;
  w.split = u / tiles;
  const int t = u - w.split * tiles;
  w.tq = t / p.tiles_p;
  w.tp = t - w.tq * p.tiles_p;
  w.kb0 = w.split * p.kb_per_split;
  w.kb1 = min(p.num_kb, w.kb0 + p.kb_per_split);
  return w;
}

// Stores the QN int32 sums of one P row: element i goes to offset
// off0 + i * step of the destination (C, or the split's partials), for the
// elements whose Q index q0 + i is inside the matrix; int32, or requantised
// to int16 / int8.  Every branch is taken per thread, outside the unrolled
// loops, so that acc stays in registers.
template <int QN>
__device__ __forceinline__ void store_row(const S8tmParams &p, const int32_t (&acc)[QN], int split, int64_t off0,
                                          int64_t step, int64_t q0) {
  const int64_t nq = p.Q_rows - q0;  // valid elements (>= 1)
  if (p.splits > 1 || p.out_bits == 32) {
    int32_t *dst = reinterpret_cast<int32_t *>(p.splits > 1 ? p.ws : p.C) +
                   (p.splits > 1 ? (int64_t)split * p.M * p.N : 0) + off0;
#pragma unroll
    for (int i = 0; i < QN; ++i)
      if (i < nq) dst[i * step] = acc[i];
  } else if (p.out_bits == 16) {
    int16_t *dst = reinterpret_cast<int16_t *>(p.C) + off0;
#pragma unroll
    for (int i = 0; i < QN; ++i)
      if (i < nq) dst[i * step] = static_cast<int16_t>(requantize_s32(acc[i], p.out_shift, -32768, 32767));
  } else {
    int8_t *dst = reinterpret_cast<int8_t *>(p.C) + off0;
#pragma unroll
    for (int i = 0; i < QN; ++i)
      if (i < nq) dst[i * step] = static_cast<int8_t>(requantize_s32(acc[i], p.out_shift, -128, 127));
  }
}

template <int QN, bool Q_KMAJOR, int STAGES, int NA>
__global__ void __launch_bounds__(kThreadsS8tm, 1)
    gemm_s8tm_kernel(const __grid_constant__ CUtensorMap tmP, const __grid_constant__ CUtensorMap tmQ,
                     const S8tmParams p) {
  using Cfg = S8tmCfg<QN, Q_KMAJOR, STAGES, NA>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-byte alignment
  uint8_t *base_ptr = smem_raw + (base - raw);
  const uint32_t sP = base + Cfg::kPOffset;
  const uint32_t sQ = base + Cfg::kQOffset;
  const uint32_t bars = base + Cfg::kBarOffset;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(base_ptr + Cfg::kBarOffset + Cfg::kNumBars * 8);
  volatile uint32_t *abort_flag = tmem_slot + 1;

  auto full_bar = [&](uint32_t s) { return bars + 8u * s; };
  auto empty_bar = [&](uint32_t s) { return bars + 8u * (STAGES + s); };
  auto pfull_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + a); };
  auto pempty_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + NA + a); };
  auto accf_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * NA + b); };
  auto acce_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * NA + 2 + b); };
  const uint32_t drain_bar = bars + 8u * (2 * STAGES + 2 * NA + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1 + kConvWarps);
    }
    for (int a = 0; a < NA; ++a) {
      mbar_init(pfull_bar(a), kConvWarps);
      mbar_init(pempty_bar(a), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), kEpiWarps * 32);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&tmP);
    tma_prefetch_desc(&tmQ);
  }
  if (warp == 1) tmem_alloc<Cfg::kTmemCols>(smem_addr(tmem_slot));
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  griddep_wait();  // the staged Q comes from the previous kernel of the stream

  const int num_units = p.tiles_p * p.tiles_q * p.splits;
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
        const S8tmUnit w = decode_s8tm(p, u);
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full_bar(s), Cfg::kStageBytes);
          tma_load_2d(sP + s * kPBytes, &tmP, kb * kKB, w.tp * kBM, full_bar(s));
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t q_dst = sQ + s * Cfg::kQBytes + h * Cfg::kQHalf;
            const int k0 = kb * kKB + h * kBK;
            if constexpr (Q_KMAJOR) {
              tma_load_2d(q_dst, &tmQ, k0, w.tq * QN, full_bar(s));
            } else {
#pragma unroll
              for (int j = 0; j < QN / 64; ++j)
                tma_load_2d(q_dst + j * (kBK * 128), &tmQ, w.tq * QN + 64 * j, k0, full_bar(s));
            }
          }
          ++g;
        }
      }
      const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
      for (uint32_t i = first; i < g; ++i) mbar_wait_drain(full_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, QN, !Q_KMAJOR);
      uint32_t g = 0, acc_cnt = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
        const S8tmUnit w = decode_s8tm(p, u);
        for (int kb_s = w.kb0; ok && kb_s < w.kb1; kb_s += p.slab_kb) {
          const int kb_e = min(w.kb1, kb_s + p.slab_kb);
          const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
          if (!mbar_wait(acce_bar(b), aph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d_tmem = tmem_base + b * QN;
          for (int kb = kb_s; kb < kb_e; ++kb) {
            const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
            const uint32_t a = g % NA, pph = (g / NA) & 1u;
            if (!mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns) ||
                !mbar_wait(pfull_bar(a), pph, abort_flag, p.err, p.wait_limit_ns)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t q0 = sQ + s * Cfg::kQBytes;
            const uint32_t a_tmem = tmem_base + Cfg::kPCol0 + a * 64;
#pragma unroll
            for (int k = 0; k < kKB / 16; ++k) {
              // one K step of 16 is 8 packed columns of the P slot; Q as B
              // in the general kernel, within the half k / 4 (K-major: 32
              // bytes along a row; MN-major: 16 K rows = 2048 bytes, 64-wide
              // chunks 8 KB apart)
              const uint32_t qh = q0 + (k >> 2) * Cfg::kQHalf, kk = k & 3;
              const uint64_t bd = Q_KMAJOR ? smem_desc_sw128(qh + kk * 32, 16, 1024)
                                           : smem_desc_sw128(qh + kk * 2048, kBK * 128, 1024);
              tc_mma_bf16_tmem_a(d_tmem, a_tmem + k * 8, bd, idesc, (kb > kb_s || k > 0) ? 1u : 0u);
            }
            tc_commit(empty_bar(s));   // the Q box may be overwritten once these MMAs finish
            tc_commit(pempty_bar(a));  // and the P slot reused
            ++g;
          }
          if (!ok) break;
          tc_commit(accf_bar(b));
          ++acc_cnt;
        }
      }
      tc_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0, kDrainNs);
    }
    __syncwarp();
  } else if (warp >= 2 + kEpiWarps) {
    // ------------------------------------------------------- converters
    // Software-pipelined by one k-block: the TMEM store of k-block g is
    // waited for (and its P slot handed to the MMA warp) only after k-block
    // g + 1 has been loaded and converted, so the store's latency overlaps
    // that work.
    const int quad = warp & 3;
    const int r = quad * 32 + lane;               // P row within the tile = TMEM lane
    const uint32_t sw = (uint32_t)r & 7u;         // 128-byte swizzle: chunk j at j ^ (r % 8)
    const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16) + Cfg::kPCol0;
    uint32_t g = 0;
    bool ok = true, pending = false;
    uint32_t pending_slot = 0;
    auto publish = [&](uint32_t slot) {  // the slot's TMEM store has landed: hand it to the MMA warp
      tmem_st_wait();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(pfull_bar(slot));
      __syncwarp();
    };
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const S8tmUnit w = decode_s8tm(p, u);
      for (int kb = w.kb0; kb < w.kb1; ++kb) {
        const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
        const uint32_t a = g % NA, pph = (g / NA) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns)) ||
            !__all_sync(0xffffffffu, mbar_wait(pempty_bar(a), pph ^ 1u, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t row = sP + s * kPBytes + (uint32_t)r * kKB;
        uint32_t o[64];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint4 v = ld_shared_v4(row + (((uint32_t)j ^ sw) << 4));  // k = 16 j .. 16 j + 15
          s8x4_to_bf16x4(v.x, o[8 * j + 0], o[8 * j + 1]);
          s8x4_to_bf16x4(v.y, o[8 * j + 2], o[8 * j + 3]);
          s8x4_to_bf16x4(v.z, o[8 * j + 4], o[8 * j + 5]);
          s8x4_to_bf16x4(v.w, o[8 * j + 6], o[8 * j + 7]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar(s));  // this warp's rows of the P box are read
        __syncwarp();
        if (pending) publish(pending_slot);
        tmem_st_32x32b_x64(lane_base + a * 64, o);
        pending = true;
        pending_slot = a;
        ++g;
      }
    }
    if (pending) publish(pending_slot);
  } else {
    // --------------------------------------------------------- epilogue
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    uint32_t acc_cnt = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const S8tmUnit w = decode_s8tm(p, u);
      int32_t acc[QN];
#pragma unroll
      for (int i = 0; i < QN; ++i) acc[i] = 0;
      for (int kb_s = w.kb0; kb_s < w.kb1; kb_s += p.slab_kb) {
        const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(accf_bar(b), aph, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t t0 = tmem_base + b * QN + ((uint32_t)(quad * 32) << 16);
#pragma unroll
        for (int c = 0; c < QN / 32; ++c) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(t0 + c * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) acc[c * 32 + i] += __float2int_rn(__uint_as_float(v[i]));
        }
        tc_fence_before_sync();
        mbar_arrive(acce_bar(b));
        ++acc_cnt;
      }
      if (!ok) break;
      const int64_t prow = (int64_t)w.tp * kBM + r;
      if (prow >= p.P_rows) continue;
      const int64_t q0 = (int64_t)w.tq * QN;
      // partials have row pitch N; C has ldc
      const int64_t ld = p.splits > 1 ? (int64_t)p.N : p.ldc;
      if (p.swap)  // C[q][prow]: per element the warp's lanes store 32 consecutive columns
        store_row<QN>(p, acc, w.split, q0 * ld + prow, ld, q0);
      else         // C[prow][q]
        store_row<QN>(p, acc, w.split, prow * ld + q0, 1, q0);
    }
  }

  griddep_launch_dependents();  // e.g. the split-K reduction may start setting up
  __syncwarp();
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after_sync();
    tmem_dealloc<Cfg::kTmemCols>(tmem_base);
  }
}

template <int QN, bool Q_KMAJOR, int STAGES, int NA>
cudaError_t launch_one(const CUtensorMap &tp, const CUtensorMap &tq, const S8tmParams &p, int grid,
                       cudaStream_t st) {
  using Cfg = S8tmCfg<QN, Q_KMAJOR, STAGES, NA>;
  auto kern = gemm_s8tm_kernel<QN, Q_KMAJOR, STAGES, NA>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_ex(kern, dim3(grid), dim3(kThreadsS8tm), Cfg::kSmemBytes, st, 1, tp, tq, p);
}

}  // namespace

cudaError_t launch_s8tm(int qn, bool q_kmajor, const CUtensorMap &tp, const CUtensorMap &tq, const S8tmParams &p,
                        int grid, cudaStream_t st) {
  // stages: 4 x 48 KB (QN 128) or 6 x 32 KB (QN 64) of operands in flight
  if (qn == 128)
    return q_kmajor ? launch_one<128, true, 4, 4>(tp, tq, p, grid, st) : launch_one<128, false, 4, 4>(tp, tq, p, grid, st);
  return q_kmajor ? launch_one<64, true, 6, 4>(tp, tq, p, grid, st) : launch_one<64, false, 6, 4>(tp, tq, p, grid, st);
}

}  // namespace gb300

// gemm_s8a.cu -- exact int8 GEMM for compute-bound 128 x 224 tiles with A
// converted to bf16 inside the kernel, into tensor memory: only B is staged.
//
// The general int8 path stages both operands as bf16 before the GEMM; at
// 4096^3 that pass moves 96 MB.  Here A stays int8 in the caller's buffer:
// TMA brings 128 x 64 int8 boxes (64-byte rows, 64-byte swizzle), four
// converter warps turn each row into 32 packed bf16 pairs and write them to
// a TMEM slot, and the MMA reads its A operand from there (tcgen05.mma with
// A in TMEM); B is staged as bf16 and read from shared memory as in the
// general kernel.  Staging B alone moves half the bytes, and the A ring's
// 8 KB stages leave room for a fifth pipeline stage.
//
// The library uses it only when GB300_GEMM_S8A=1: it is exact, but on GB300
// int8 4096^3 took 151 us against 110 us for staging both operands.  With
// two A slots, and the converters publishing a slot one k-block late, the
// MMAs of k-block g wait for those of k-block g - 1 to complete.
//
// TMEM holds the two 224-column fp32 accumulators and two 32-column A slots
// (512 columns).  The 16 warps split the register file with setmaxnreg:
//   warpgroup 0 (56 registers)  warp 0 lane 0 TMA producer, warp 1 lane 0
//                               MMA issuer (and TMEM allocation); warps 2-3
//                               idle
//   warpgroup 1 (80)            converters, one per TMEM lane quadrant
//   warpgroups 2-3 (184)        the int8 epilogue of the general kernel:
//                               eight warps, 112 int32 sums per thread
// 128 x 56 + 128 x 80 + 256 x 184 = 64512 of the 65536 registers the block
// is launched with (512 threads x 128).
//
// Exactness is the general int8 path's: the MMA warp closes the accumulator
// every 16 k-blocks (1024 K elements), each slab's fp32 sums are integers
// below 2^24 in magnitude and exact, and the epilogue adds them in int32.
#include <cuda_bf16.h>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kS8aThreads = 512;
constexpr uint32_t kAI8Bytes = kBM * 64;  // 128 rows x 64 int8

template <int BN, int STAGES, int NA>
struct S8aCfg {
  static constexpr int kEpiWarps = 8;
  static constexpr int kCPT = BN / 2;  // columns per epilogue thread
  static constexpr uint32_t kBBytes = BN * kRowBytes;
  static constexpr uint32_t kAOff = 0;
  static constexpr uint32_t kBOff = STAGES * kAI8Bytes;             // 1024-byte aligned
  static constexpr uint32_t kEpiOff = kBOff + STAGES * kBBytes;     // 1024-byte aligned
  static constexpr uint32_t kBarOff = kEpiOff + kEpiWarps * 4096u;  // one 4 KB staging block per epilogue warp
  static constexpr uint32_t kNumBars = 2 * STAGES + 2 * NA + 5;
  static constexpr uint32_t kSmemBytes = kBarOff + kNumBars * 8 + 16 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA is 227 KB");
  static constexpr uint32_t kACol0 = 2 * BN;  // A slots (32 columns each) follow the accumulators
  static constexpr uint32_t kTmemCols = pow2_at_least(2 * BN + 32 * NA);
  static_assert(kTmemCols <= 512, "TMEM has 512 columns");
  static_assert(kCPT % 32 == 16, "the epilogue moves 32-column chunks and one of 16");
};

template <int BN, int STAGES, int NA>
__global__ void __launch_bounds__(kS8aThreads, 1)
    gemm_s8a_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmOut, const TcParams p) {
  using Cfg = S8aCfg<BN, STAGES, NA>;
  constexpr int CPT = Cfg::kCPT;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *base_ptr = smem_raw + (base - raw);
  const uint32_t sA = base + Cfg::kAOff;
  const uint32_t sB = base + Cfg::kBOff;
  const uint32_t bars = base + Cfg::kBarOff;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(base_ptr + Cfg::kBarOff + Cfg::kNumBars * 8);
  volatile uint32_t *abort_flag = tmem_slot + 1;

  auto full_bar = [&](uint32_t s) { return bars + 8u * s; };
  auto empty_bar = [&](uint32_t s) { return bars + 8u * (STAGES + s); };
  auto tfull_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + a); };
  auto tempty_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + NA + a); };
  auto accf_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * NA + b); };
  auto acce_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * NA + 2 + b); };
  const uint32_t drain_bar = bars + 8u * (2 * STAGES + 2 * NA + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int wg = warp >> 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1 + 4);  // the MMAs' commit (B) and the four converter warps (A)
    }
    for (int a = 0; a < NA; ++a) {
      mbar_init(tfull_bar(a), 4);
      mbar_init(tempty_bar(a), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), Cfg::kEpiWarps * 32);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (p.out_tma != kOutDirect) tma_prefetch_desc(&tmOut);
  }
  if (warp == 1) tmem_alloc<Cfg::kTmemCols>(smem_addr(tmem_slot));
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  griddep_wait();  // B is staged by the previous kernel of the stream

  const int num_units = p.tiles_m * p.tiles_n;
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

  if (wg == 0) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 56;" ::: "memory");
    if (warp == 0 && lane == 0) {
      // ------------------------------------------------------ TMA producer
      uint32_t g = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
        const Unit w = decode_unit(p, u);
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full_bar(s), kAI8Bytes + Cfg::kBBytes);
          tma_load_2d(sA + s * kAI8Bytes, &tmA, kb * kBK, w.tm * kBM, full_bar(s));
          tma_load_2d(sB + s * Cfg::kBBytes, &tmB, kb * kBK, w.tn * BN, full_bar(s));
          ++g;
        }
      }
      const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
      for (uint32_t i = first; i < g; ++i) mbar_wait_drain(full_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
    } else if (warp == 1 && lane == 0) {
      // ------------------------------------------------------- MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, BN, false);
      uint32_t g = 0, acc_cnt = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
        const Unit w = decode_unit(p, u);
        for (int kb_s = w.kb0; ok && kb_s < w.kb1; kb_s += p.slab_kb) {
          const int kb_e = min(w.kb1, kb_s + p.slab_kb);
          const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
          if (!mbar_wait(acce_bar(b), aph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d_tmem = tmem_base + b * BN;
          for (int kb = kb_s; kb < kb_e; ++kb) {
            const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
            const uint32_t a = g % NA, tph = (g / NA) & 1u;
            if (!mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns) ||
                !mbar_wait(tfull_bar(a), tph, abort_flag, p.err, p.wait_limit_ns)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t b0 = sB + s * Cfg::kBBytes;
            const uint32_t a_tmem = tmem_base + Cfg::kACol0 + a * 32;
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              tc_mma_bf16_tmem_a(d_tmem, a_tmem + k * 8, smem_desc_sw128(b0 + k * 32, 16, 1024), idesc,
                                 (kb > kb_s || k > 0) ? 1u : 0u);
            tc_commit(empty_bar(s));   // B's stage may be refilled once these MMAs finish
            tc_commit(tempty_bar(a));  // and the A slot reused
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
  } else if (wg == 1) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 80;" ::: "memory");
    // ------------------------------------------------------- converters
    // Pipelined by one k-block: the TMEM store of k-block g is published to
    // the MMA warp after k-block g + 1 has been converted.
    const int quad = warp & 3;
    const int r = quad * 32 + lane;               // A row within the tile = TMEM lane
    const uint32_t sw = ((uint32_t)r >> 1) & 3u;  // 64-byte swizzle: chunk j at j ^ ((r / 2) % 4)
    const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16) + Cfg::kACol0;
    uint32_t g = 0;
    bool ok = true, pending = false;
    uint32_t pending_slot = 0;
    auto publish = [&](uint32_t slot) {
      tmem_st_wait();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(tfull_bar(slot));
      __syncwarp();
    };
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      for (int kb = w.kb0; kb < w.kb1; ++kb) {
        const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
        const uint32_t a = g % NA, tph = (g / NA) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns)) ||
            !__all_sync(0xffffffffu, mbar_wait(tempty_bar(a), tph ^ 1u, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t row = sA + s * kAI8Bytes + (uint32_t)r * 64u;
        uint32_t o[32];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint4 v = ld_shared_v4(row + (((uint32_t)j ^ sw) << 4));  // k = 16 j .. 16 j + 15
          s8x4_to_bf16x4(v.x, o[8 * j + 0], o[8 * j + 1]);
          s8x4_to_bf16x4(v.y, o[8 * j + 2], o[8 * j + 3]);
          s8x4_to_bf16x4(v.z, o[8 * j + 4], o[8 * j + 5]);
          s8x4_to_bf16x4(v.w, o[8 * j + 6], o[8 * j + 7]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar(s));  // this warp's rows of the A box are read
        __syncwarp();
        if (pending) publish(pending_slot);
        tmem_st_32x32b_x32(lane_base + a * 32, o);
        pending = true;
        pending_slot = a;
        ++g;
      }
    }
    if (pending) publish(pending_slot);
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 184;" ::: "memory");
    // --------------------------------------------------------- epilogue
    const int ew = warp - 8;
    const int quad = warp & 3;
    const int colpart = ew >> 2;
    const int row_in_tile = quad * 32 + lane;
    const uint32_t ebuf = base + Cfg::kEpiOff + ew * 4096u;
    uint32_t acc_cnt = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      const int64_t row = (int64_t)w.tm * kBM + row_in_tile;
      const bool row_ok = row < p.M;
      const int col0 = w.tn * BN + colpart * CPT;
      const int y0 = w.tm * kBM + quad * 32;
      int32_t acc[CPT];
#pragma unroll
      for (int i = 0; i < CPT; ++i) acc[i] = 0;
      for (int kb_s = w.kb0; kb_s < w.kb1; kb_s += p.slab_kb) {
        const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(accf_bar(b), aph, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t t0 = tmem_base + b * BN + ((uint32_t)(quad * 32) << 16) + colpart * CPT;
#pragma unroll
        for (int c = 0; c < CPT / 32; ++c) {
          uint32_t r[32];
          tmem_ld_32x32b_x32(t0 + c * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) acc[c * 32 + i] += __float2int_rn(__uint_as_float(r[i]));
        }
        {
          constexpr int kTail = (CPT / 32) * 32;
          uint32_t r[16];
          tmem_ld_32x32b_x16(t0 + kTail, r);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[kTail + i] += __float2int_rn(__uint_as_float(r[i]));
        }
        tc_fence_before_sync();
        mbar_arrive(acce_bar(b));
        ++acc_cnt;
      }
      if (!ok) break;
      if (p.out_tma == kOutTmaC) {
#pragma unroll
        for (int c = 0; c < CPT / 32; ++c) {
          uint32_t v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = static_cast<uint32_t>(acc[c * 32 + i]);
          const int x = col0 + c * 32;
          if (p.out_bits == 32)
            tma_out_words32<false>(&tmOut, ebuf, lane, v, x, y0, 0, y0 < p.M && x < p.N);
          else
            tma_out_narrow(&tmOut, ebuf, lane, v, p.out_bits, p.out_shift, x, y0, y0 < p.M && x < p.N);
        }
      } else if (row_ok) {
#pragma unroll
        for (int c = 0; c < CPT / 32; ++c) {
          uint32_t v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = static_cast<uint32_t>(acc[c * 32 + i]);
          store_s8_result<32>(p, row, col0 + c * 32, v);
        }
      }
      if (row_ok) {  // the 16-column tail: each lane stores its row
        constexpr int kTail = (CPT / 32) * 32;
        uint32_t v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = static_cast<uint32_t>(acc[kTail + i]);
        store_s8_result<16>(p, row, col0 + kTail, v);
      }
    }
    if (lane == 0) bulk_wait_all();  // this warp's TMA stores have landed
  }

  griddep_launch_dependents();
  __syncwarp();
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after_sync();
    tmem_dealloc<Cfg::kTmemCols>(tmem_base);
  }
}

}  // namespace

cudaError_t launch_s8a(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o, const TcParams &p, int grid,
                       cudaStream_t st) {
  using Cfg = S8aCfg<224, 5, 2>;
  auto kern = gemm_s8a_kernel<224, 5, 2>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_ex(kern, dim3((unsigned)grid), dim3(kS8aThreads), Cfg::kSmemBytes, st, 1, a, b, o, p);
}

}  // namespace gb300

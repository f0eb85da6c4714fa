// gemm_s8x.cu -- exact int8 GEMM on the tensor cores with both operands
// converted inside the kernel: no staging launch, no 16-bit copies in HBM.
//
// The general int8 path stages A and B as bf16 in a launch of its own: three
// bytes of HBM traffic per operand element, about 17 us of a 112 us GEMM at
// 4096^3.  Here both operands stay int8 in the caller's buffers.  For every
// 64-deep K step the TMA brings a 128 x 64 int8 box of A and a BN x 64 int8
// box of B (64-byte rows, 64-byte swizzle) into a ring, and converter warps
// turn them into fp16 -- every int8 value is exact in fp16, and a byte
// permute plus a packed subtraction convert two of them (s8x4_to_f16x4):
//   A into one of two 32-column TMEM slots, the MMA's A operand read from
//     tensor memory (TMEM lane = row of the tile);
//   B into one of NB fp16 tiles in shared memory, laid out as the MMA's
//     K-major, 128-byte-swizzled B operand.
// The MMA is tcgen05.mma kind::f16 with fp16 A and B and fp32 accumulation,
// closed every 16 K steps (1024 products of magnitude <= 2^14: every partial
// sum is an integer below 2^24, exact in fp32) and drained into int32 sums
// by the epilogue, as in the general int8 kernel.  Shared-memory traffic per
// K step (int8 boxes written and read, the fp16 B tile written and read by
// the MMA) stays close to the bf16 kernel's, which is what converting both
// operands in shared memory could not do.
//
// Warps (512 threads; registers redistributed with setmaxnreg):
//   0        TMA producer (lane 0)                   warpgroup 0: 64 registers
//   1        MMA issuer (lane 0); TMEM allocation
//   2, 3     B converters (8 of B's 16-byte pieces per lane and K step)
//   4 - 7    A converters -- warp w converts the 32 rows of TMEM lanes
//            32 (w % 4) .. -- and then a few B pieces  warpgroup 1: 80
//   8 - 15   epilogue: 112 int32 sums per thread      warpgroups 2, 3: 184
// 128 x 64 + 128 x 80 + 256 x 184 = 65536: the registers the block is
// launched with (512 threads x 128).
#include <type_traits>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kS8xThreads = 512;
constexpr int kS8xConvWarps = 6;
constexpr int kS8xNA = 2;                 // A slots in TMEM (32 columns each)
constexpr uint32_t kAI8Bytes = kBM * 64;  // 128 rows x 64 int8

template <int BN, int STAGES, int NB>
struct S8xCfg {
  static_assert(BN > 128 && BN <= 256 && (BN - 128) % 32 == 0, "B pieces split 8 / (BN - 128) / 32 per lane");
  static constexpr int kEpiWarps = 8;
  static constexpr int kCPT = BN / 2;                  // columns per epilogue thread
  static_assert(kCPT % 16 == 0, "the epilogue moves 32-column chunks and one of 16");
  static constexpr uint32_t kBI8Bytes = BN * 64u;      // BN rows x 64 int8
  static constexpr uint32_t kBH16Bytes = BN * 128u;    // BN rows x 64 fp16
  static constexpr uint32_t kAOff = 0;
  static constexpr uint32_t kBOff = STAGES * kAI8Bytes;                // 1024-byte aligned
  static constexpr uint32_t kHOff = kBOff + STAGES * kBI8Bytes;        // 1024-byte aligned (BN % 16 == 0)
  static constexpr uint32_t kEpiOff = kHOff + NB * kBH16Bytes;
  static constexpr uint32_t kBarOff = kEpiOff + kEpiWarps * 4096u;     // one 4 KB staging block per epilogue warp
  static constexpr uint32_t kNumBars = 2 * STAGES + 2 * kS8xNA + 2 * NB + 5;
  static constexpr uint32_t kSmemBytes = kBarOff + kNumBars * 8 + 16 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA is 227 KB");
  static constexpr uint32_t kACol0 = 2 * BN;           // A slots follow the two accumulators
  static constexpr uint32_t kTmemCols = pow2_at_least(2 * BN + 32 * kS8xNA);
  static_assert(kTmemCols <= 512, "TMEM has 512 columns");
};

template <int BN, int STAGES, int NB>
__global__ void __launch_bounds__(kS8xThreads, 1)
    gemm_s8x_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmOut, const TcParams p) {
  using Cfg = S8xCfg<BN, STAGES, NB>;
  constexpr int CPT = Cfg::kCPT;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *base_ptr = smem_raw + (base - raw);
  const uint32_t sA = base + Cfg::kAOff;   // int8 A boxes
  const uint32_t sB = base + Cfg::kBOff;   // int8 B boxes
  const uint32_t sH = base + Cfg::kHOff;   // fp16 B tiles
  const uint32_t bars = base + Cfg::kBarOff;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(base_ptr + Cfg::kBarOff + Cfg::kNumBars * 8);
  volatile uint32_t *abort_flag = tmem_slot + 1;

  auto full_bar = [&](uint32_t s) { return bars + 8u * s; };                 // int8 boxes landed
  auto empty_bar = [&](uint32_t s) { return bars + 8u * (STAGES + s); };     // int8 boxes read
  auto tfull_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + a); }; // A slot written
  auto tempty_bar = [&](uint32_t a) { return bars + 8u * (2 * STAGES + kS8xNA + a); };
  auto hfull_bar = [&](uint32_t t) { return bars + 8u * (2 * STAGES + 2 * kS8xNA + t); };  // fp16 B tile written
  auto hempty_bar = [&](uint32_t t) { return bars + 8u * (2 * STAGES + 2 * kS8xNA + NB + t); };
  auto accf_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * kS8xNA + 2 * NB + b); };
  auto acce_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 * kS8xNA + 2 * NB + 2 + b); };
  const uint32_t drain_bar = bars + 8u * (2 * STAGES + 2 * kS8xNA + 2 * NB + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int wg = warp >> 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), kS8xConvWarps);
    }
    for (int a = 0; a < kS8xNA; ++a) {
      mbar_init(tfull_bar(a), 4);
      mbar_init(tempty_bar(a), 1);
    }
    for (int t = 0; t < NB; ++t) {
      mbar_init(hfull_bar(t), kS8xConvWarps);
      mbar_init(hempty_bar(t), 1);
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
  // A and B may be written by the previous kernel of the stream.
  griddep_wait();

  const int num_units = p.tiles_m * p.tiles_n;
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

  // The converter loop, one copy per role, each compiled within its
  // warpgroup's register budget (64 for warps 2, 3; 80 for warps 4-7).
  auto convert = [&](auto role) {
    // ------------------------------------------------------- converters
    constexpr bool a_role = decltype(role)::value;
    const int cw = warp - 2;                      // 0, 1: B only; 2..5: A, then B
    const int quad = warp & 3;
    const int r = quad * 32 + lane;               // A row within the tile = TMEM lane
    const uint32_t sw = ((uint32_t)r >> 1) & 3u;  // 64-byte swizzle: chunk j of row r at j ^ ((r / 2) % 4)
    const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16) + Cfg::kACol0;
    // B pieces (16 int8 of one row: piece i is row i / 4, k 16 (i % 4) ..):
    // warps 2, 3 take 256 each, warps 4..7 BN - 128 each; 32 consecutive
    // pieces of a warp are 8 whole rows, so the reads and writes of a warp
    // instruction cover distinct bank groups.
    const int it0 = a_role ? 512 + (cw - 2) * (BN - 128) : cw * 256;
    constexpr int kItA = (BN - 128) / 32, kItB = 8;
    uint32_t g = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      for (int kb = w.kb0; kb < w.kb1; ++kb) {
        const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
        const uint32_t a = g % kS8xNA, tph = (g / kS8xNA) & 1u;
        const uint32_t t = g % NB, hph = (g / NB) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        if constexpr (a_role) {
          if (!__all_sync(0xffffffffu, mbar_wait(tempty_bar(a), tph ^ 1u, abort_flag, p.err, p.wait_limit_ns))) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t row = sA + s * kAI8Bytes + (uint32_t)r * 64u;
          uint32_t o[32];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 v = ld_shared_v4(row + (((uint32_t)j ^ sw) << 4));  // k = 16 j .. 16 j + 15
            s8x4_to_f16x4(v.x, o[8 * j + 0], o[8 * j + 1]);
            s8x4_to_f16x4(v.y, o[8 * j + 2], o[8 * j + 3]);
            s8x4_to_f16x4(v.z, o[8 * j + 4], o[8 * j + 5]);
            s8x4_to_f16x4(v.w, o[8 * j + 6], o[8 * j + 7]);
          }
          tmem_st_32x32b_x32(lane_base + a * 32, o);
          tmem_st_wait();
          tc_fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(tfull_bar(a));  // the MMA may read the slot
        }
        if (!__all_sync(0xffffffffu, mbar_wait(hempty_bar(t), hph ^ 1u, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        const uint32_t src = sB + s * Cfg::kBI8Bytes, dst = sH + t * Cfg::kBH16Bytes;
        const int nit = a_role ? kItA : kItB;
#pragma unroll 4
        for (int i = 0; i < nit; ++i) {
          const int it = it0 + i * 32 + lane;
          const uint32_t n = (uint32_t)it >> 2, j = (uint32_t)it & 3u;
          const uint4 v = ld_shared_v4(src + n * 64u + ((j ^ ((n >> 1) & 3u)) << 4));
          uint32_t h[8];
          s8x4_to_f16x4(v.x, h[0], h[1]);
          s8x4_to_f16x4(v.y, h[2], h[3]);
          s8x4_to_f16x4(v.z, h[4], h[5]);
          s8x4_to_f16x4(v.w, h[6], h[7]);
          // fp16 row n: 16-byte chunk c (k 8c .. 8c + 7) at c ^ (n % 8)
          const uint32_t drow = dst + n * 128u, x = n & 7u;
          st_shared_v4(drow + (((2u * j) ^ x) << 4), h[0], h[1], h[2], h[3]);
          st_shared_v4(drow + (((2u * j + 1u) ^ x) << 4), h[4], h[5], h[6], h[7]);
        }
        fence_proxy_async_smem();  // the generic-proxy writes, before the MMA reads them
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(empty_bar(s));  // this warp is done with the int8 boxes
          mbar_arrive(hfull_bar(t));
        }
        __syncwarp();
        ++g;
      }
    }
  };

  if (wg == 0) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 64;" ::: "memory");
    if (warp == 0) {
      // ------------------------------------------------------ TMA producer
      if (lane == 0) {
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
            mbar_arrive_expect_tx(full_bar(s), kAI8Bytes + Cfg::kBI8Bytes);
            tma_load_2d(sA + s * kAI8Bytes, &tmA, kb * kBK, w.tm * kBM, full_bar(s));
            tma_load_2d(sB + s * Cfg::kBI8Bytes, &tmB, kb * kBK, w.tn * BN, full_bar(s));
            ++g;
          }
        }
        // every load this thread issued has landed before the CTA may exit
        const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
        for (uint32_t i = first; i < g; ++i) mbar_wait_drain(full_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
      }
      __syncwarp();
    } else if (warp == 1) {
      // ------------------------------------------------------- MMA issuer
      if (lane == 0) {
        constexpr uint32_t idesc = idesc_f16_f32(kBM, BN);
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
              const uint32_t a = g % kS8xNA, tph = (g / kS8xNA) & 1u;
              const uint32_t t = g % NB, hph = (g / NB) & 1u;
              if (!mbar_wait(tfull_bar(a), tph, abort_flag, p.err, p.wait_limit_ns) ||
                  !mbar_wait(hfull_bar(t), hph, abort_flag, p.err, p.wait_limit_ns)) {
                ok = false;
                break;
              }
              tc_fence_after_sync();
              const uint32_t a_tmem = tmem_base + Cfg::kACol0 + a * 32;
              const uint32_t b0 = sH + t * Cfg::kBH16Bytes;
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                tc_mma_bf16_tmem_a(d_tmem, a_tmem + k * 8, smem_desc_sw128(b0 + k * 32, 16, 1024), idesc,
                                   (kb > kb_s || k > 0) ? 1u : 0u);
              tc_commit(tempty_bar(a));  // the A slot and
              tc_commit(hempty_bar(t));  // the fp16 B tile may be rewritten once these MMAs finish
              ++g;
            }
            if (!ok) break;
            tc_commit(accf_bar(b));  // the slab's sums are ready for the epilogue
            ++acc_cnt;
          }
        }
        tc_commit(drain_bar);  // all MMAs complete before TMEM is released
        mbar_wait_drain(drain_bar, 0, kDrainNs);
      }
      __syncwarp();
    } else {
      convert(std::false_type{});  // warps 2, 3: B only
    }
  } else if (wg == 1) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 80;" ::: "memory");
    convert(std::true_type{});  // A, then B
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
          uint32_t rr[32];
          tmem_ld_32x32b_x32(t0 + c * 32, rr);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) acc[c * 32 + i] += __float2int_rn(__uint_as_float(rr[i]));
        }
        if constexpr (CPT % 32 != 0) {
          constexpr int kTail = (CPT / 32) * 32;
          uint32_t rr[16];
          tmem_ld_32x32b_x16(t0 + kTail, rr);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[kTail + i] += __float2int_rn(__uint_as_float(rr[i]));
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
      if constexpr (CPT % 32 != 0) {
        if (row_ok) {  // the 16-column tail: each lane stores its row
          constexpr int kTail = (CPT / 32) * 32;
          uint32_t v[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = static_cast<uint32_t>(acc[kTail + i]);
          store_s8_result<16>(p, row, col0 + kTail, v);
        }
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

cudaError_t launch_s8x(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o, const TcParams &p, int grid,
                       cudaStream_t st) {
  constexpr int kBN = kS8xBN, kStages = kS8xStages, kNB = 3;
  using Cfg = S8xCfg<kBN, kStages, kNB>;
  auto kern = gemm_s8x_kernel<kBN, kStages, kNB>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_ex(kern, dim3((unsigned)grid), dim3(kS8xThreads), Cfg::kSmemBytes, st, 1, a, b, o, p);
}

}  // namespace gb300

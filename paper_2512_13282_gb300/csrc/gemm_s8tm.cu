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
//   P  the large operand, int8: B when M is small (P row = column n of C),
//      or A when N is small (P row = row m).  It is the MMA's 128-row A
//      operand, read from TMEM.  P is either K contiguous (A, or B stored
//      N x K) or P row contiguous (B stored K x N: the TMA box then holds
//      128 k-rows of 128 P rows, and the converters read it transposed).
//   Q  the small operand, staged beforehand (s8tm_stage_q_kernel) as the
//      exact shared-memory image the MMA reads for each (Q tile, k-block):
//      bf16, K-major, 128-byte swizzled, QN rows x 128 K = QN x 256 bytes,
//      contiguous; zero outside the matrix.  It is the MMA's QN-column B
//      operand.
//
// Roles (11 warps):
//   warp 0 (one lane)  P producer: per k-block of 128 a 128 x 128 int8 TMA
//                      box of P (128-byte rows, 128-byte swizzle) into a
//                      deep ring of its own.  Every row of a TMA box is a
//                      request of its own; 128-byte rows move twice the
//                      bytes per request of 64-byte ones (measured on
//                      GB300: twice the bytes per second per SM).
//   warp 10 (one lane) Q producer: Q's image with one bulk copy into a
//                      shallow ring (Q is read from L2).
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
// every 8 k-blocks of 128 (1024 K elements) and the epilogue converts each
// slab to int32 (exactly) and adds the slabs in int32 registers.
//
// A P stage is free again once every converter warp has read its rows (one
// arrival per warp), a Q stage once the MMAs that read it have completed
// (tcgen05.commit), a TMEM P slot likewise.  With P decoupled from the MMA,
// the P ring keeps its boxes in flight from HBM: measured on GB300, a P box
// takes about 2 us from issue to arrival under load, so the bytes in flight
// per SM, not the converters or the MMAs, set the stream rate.
#include <cuda_bf16.h>

#include "gemm_internal.h"

namespace gb300 {

namespace {

constexpr int kConvWarps = 4;
constexpr int kEpiWarps = 4;
constexpr int kQWarp = 2 + kEpiWarps + kConvWarps;                // 10: Q producer
constexpr int kThreadsS8tm = (kQWarp + 1) * 32;                   // 352
constexpr int kKB = kS8tmKB;                                      // K per k-block
constexpr uint32_t kPBytes = kBM * kKB;                           // 128 rows x 128 int8

// SP stages of P (16 KB each) and SQ of Q (QN x 256 bytes each) in two
// separate rings: a P stage is free again as soon as the converters have
// read it, so the P ring keeps SP boxes in flight from HBM whatever the MMA
// does; Q comes from L2 and needs only a few stages.
template <int QN, int SP, int SQ, int NA>
struct S8tmCfg {
  static_assert(QN == 64 || QN == 128, "QN is 64 or 128");
  static constexpr uint32_t kQHalf = QN * kRowBytes;  // QN x 64 bf16: one half of a Q image
  static constexpr uint32_t kQBytes = 2 * kQHalf;      // the k-block's Q image
  static constexpr uint32_t kPOffset = 0;
  static constexpr uint32_t kQOffset = SP * kPBytes;  // 1024-byte aligned
  // one 32 x 32 int32 block per epilogue warp, staging the TMA reductions
  // of split-K into C (128-byte swizzle; 1024-byte aligned)
  static constexpr uint32_t kEpiOffset = kQOffset + SQ * kQBytes;
  static constexpr uint32_t kBarOffset = kEpiOffset + kEpiWarps * 4096;
  static constexpr uint32_t kNumBars = 2 * SP + 2 * SQ + 2 * NA + 5;
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
  if (p.add_into_c) {
    // int32 C, zeroed by the Q staging kernel: every split adds its exact
    // partial sums (integer addition, so any order gives the same C), here
    // element by element where C's alignment rules out TMA reductions
    int32_t *dst = reinterpret_cast<int32_t *>(p.C) + off0;
#pragma unroll
    for (int i = 0; i < QN; ++i)
      if (i < nq) atomicAdd(dst + i * step, acc[i]);
  } else if (p.splits > 1 || p.out_bits == 32) {
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

// Split-K of int32 C with TMA reductions: the warp's QN sums of its 32 P
// rows, 32 Q columns at a time, staged as a 32 x 32 block (128-byte rows,
// 16-byte chunk j of row r at chunk j ^ (r % 8)) and added into C by one TMA
// reduction (element-wise atomic; the TMA clips a block that crosses C's
// edges, and a block that starts outside C is not issued).  C[q][prow]
// (swap): block row = q, column = lane; else C[prow][q]: row = lane.
template <int QN>
__device__ __forceinline__ void reduce_rows_tma(const CUtensorMap *tm, uint32_t buf, int lane, const int32_t (&acc)[QN],
                                                bool swap, int32_t prow0, int32_t q0, int32_t P_rows, int32_t Q_rows) {
#pragma unroll
  for (int c = 0; c < QN / 32; ++c) {
    if (lane == 0) bulk_wait_read_all();  // the previous reduction has read the block
    __syncwarp();
    if (swap) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        st_shared_u32(buf + i * 128 + ((((uint32_t)lane >> 2) ^ ((uint32_t)i & 7u)) << 4) + ((uint32_t)lane & 3u) * 4,
                      static_cast<uint32_t>(acc[c * 32 + i]));
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        st_shared_v4(buf + lane * 128 + (((uint32_t)j ^ ((uint32_t)lane & 7u)) << 4),
                     static_cast<uint32_t>(acc[c * 32 + 4 * j]), static_cast<uint32_t>(acc[c * 32 + 4 * j + 1]),
                     static_cast<uint32_t>(acc[c * 32 + 4 * j + 2]), static_cast<uint32_t>(acc[c * 32 + 4 * j + 3]));
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0 && prow0 < P_rows && q0 + c * 32 < Q_rows) {
      if (swap)
        tma_reduce_add_2d(tm, buf, prow0, q0 + c * 32);
      else
        tma_reduce_add_2d(tm, buf, q0 + c * 32, prow0);
      bulk_commit();
    }
  }
}

template <int QN, int SP, int SQ, int NA, bool PK>
__global__ void __launch_bounds__(kThreadsS8tm, 1)
    gemm_s8tm_kernel(const __grid_constant__ CUtensorMap tmP, const __grid_constant__ CUtensorMap tmC,
                     const S8tmParams p) {
  using Cfg = S8tmCfg<QN, SP, SQ, NA>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-byte alignment
  uint8_t *base_ptr = smem_raw + (base - raw);
  const uint32_t sP = base + Cfg::kPOffset;
  const uint32_t sQ = base + Cfg::kQOffset;
  const uint32_t bars = base + Cfg::kBarOffset;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(base_ptr + Cfg::kBarOffset + Cfg::kNumBars * 8);
  volatile uint32_t *abort_flag = tmem_slot + 1;

  // P ring, Q ring, TMEM P slots, accumulators
  auto pfull_bar = [&](uint32_t s) { return bars + 8u * s; };
  auto pempty_bar = [&](uint32_t s) { return bars + 8u * (SP + s); };
  auto qfull_bar = [&](uint32_t s) { return bars + 8u * (2 * SP + s); };
  auto qempty_bar = [&](uint32_t s) { return bars + 8u * (2 * SP + SQ + s); };
  auto tfull_bar = [&](uint32_t a) { return bars + 8u * (2 * SP + 2 * SQ + a); };
  auto tempty_bar = [&](uint32_t a) { return bars + 8u * (2 * SP + 2 * SQ + NA + a); };
  auto accf_bar = [&](uint32_t b) { return bars + 8u * (2 * SP + 2 * SQ + 2 * NA + b); };
  auto acce_bar = [&](uint32_t b) { return bars + 8u * (2 * SP + 2 * SQ + 2 * NA + 2 + b); };
  const uint32_t drain_bar = bars + 8u * (2 * SP + 2 * SQ + 2 * NA + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < SP; ++s) {
      mbar_init(pfull_bar(s), 1);
      mbar_init(pempty_bar(s), kConvWarps);
    }
    for (int s = 0; s < SQ; ++s) {
      mbar_init(qfull_bar(s), 1);
      mbar_init(qempty_bar(s), 1);
    }
    for (int a = 0; a < NA; ++a) {
      mbar_init(tfull_bar(a), kConvWarps);
      mbar_init(tempty_bar(a), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), kEpiWarps * 32);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&tmP);
    if (p.c_tma) tma_prefetch_desc(&tmC);
  }
  if (warp == 1) tmem_alloc<Cfg::kTmemCols>(smem_addr(tmem_slot));
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  // The previous kernel of the stream is the Q staging launch (a plain
  // launch: everything before it on the stream completed before it began).
  // It writes Q's images and, for split-K into int32 C, zeroes C: the Q
  // producer and the epilogue wait for it (griddep_wait) before touching
  // those, while P, written before the staging launch began, is streamed at
  // once, so that the P ring fills while the staging kernel still runs.

  const int num_units = p.tiles_p * p.tiles_q * p.splits;
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

  if (warp == 0 || warp == kQWarp) {
    // -------------------------------------------- producers (P, then Q)
    if (lane == 0) {
      const bool is_p = warp == 0;
      if (!is_p) griddep_wait();
      const int ns = is_p ? SP : SQ;
      uint32_t g = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
        const S8tmUnit w = decode_s8tm(p, u);
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          const uint32_t s = g % ns, ph = (g / ns) & 1u;
          if (!mbar_wait(is_p ? pempty_bar(s) : qempty_bar(s), ph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          if (is_p) {
            mbar_arrive_expect_tx(pfull_bar(s), kPBytes);
            if constexpr (PK)
              tma_load_2d(sP + s * kPBytes, &tmP, kb * kKB, w.tp * kBM, pfull_bar(s));
            else
              tma_load_2d(sP + s * kPBytes, &tmP, w.tp * kBM, kb * kKB, pfull_bar(s));
          } else {
            mbar_arrive_expect_tx(qfull_bar(s), Cfg::kQBytes);
            const uint8_t *q_src = static_cast<const uint8_t *>(p.q_img) +
                                   ((int64_t)w.tq * p.num_kb + kb) * (int64_t)Cfg::kQBytes;
            bulk_load(sQ + s * Cfg::kQBytes, q_src, Cfg::kQBytes, qfull_bar(s));
          }
          ++g;
        }
      }
      // Every copy this thread issued has landed before the CTA may exit.
      const uint32_t first = g > (uint32_t)ns ? g - ns : 0u;
      for (uint32_t i = first; i < g; ++i)
        mbar_wait_drain(is_p ? pfull_bar(i % ns) : qfull_bar(i % ns), (i / ns) & 1u, kDrainNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, QN, false);
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
            const uint32_t s = g % SQ, ph = (g / SQ) & 1u;
            const uint32_t a = g % NA, tph = (g / NA) & 1u;
            if (!mbar_wait(qfull_bar(s), ph, abort_flag, p.err, p.wait_limit_ns) ||
                !mbar_wait(tfull_bar(a), tph, abort_flag, p.err, p.wait_limit_ns)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t q0 = sQ + s * Cfg::kQBytes;
            const uint32_t a_tmem = tmem_base + Cfg::kPCol0 + a * 64;
#pragma unroll
            for (int k = 0; k < kKB / 16; ++k) {
              // one K step of 16 is 8 packed columns of the P slot, and 32
              // bytes along the rows of Q's half k / 4 (K-major, 128-byte
              // swizzle, 8-row atoms 1024 bytes apart)
              const uint32_t qh = q0 + (k >> 2) * Cfg::kQHalf, kk = k & 3;
              const uint64_t bd = smem_desc_sw128(qh + kk * 32, 16, 1024);
              tc_mma_bf16_tmem_a(d_tmem, a_tmem + k * 8, bd, idesc, (kb > kb_s || k > 0) ? 1u : 0u);
            }
            tc_commit(qempty_bar(s));  // the Q stage may be refilled once these MMAs finish
            tc_commit(tempty_bar(a));  // and the P slot reused
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
      if (lane == 0) mbar_arrive(tfull_bar(slot));
      __syncwarp();
    };
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const S8tmUnit w = decode_s8tm(p, u);
      for (int kb = w.kb0; kb < w.kb1; ++kb) {
        const uint32_t s = g % SP, ph = (g / SP) & 1u;
        const uint32_t a = g % NA, tph = (g / NA) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(pfull_bar(s), ph, abort_flag, p.err, p.wait_limit_ns)) ||
            !__all_sync(0xffffffffu, mbar_wait(tempty_bar(a), tph ^ 1u, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        uint32_t o[64];  // o[c]: bf16 of k = 2c (low half) and 2c + 1
        if constexpr (PK) {
          const uint32_t row = sP + s * kPBytes + (uint32_t)r * kKB;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const uint4 v = ld_shared_v4(row + (((uint32_t)j ^ sw) << 4));  // k = 16 j .. 16 j + 15
            s8x4_to_bf16x4(v.x, o[8 * j + 0], o[8 * j + 1]);
            s8x4_to_bf16x4(v.y, o[8 * j + 2], o[8 * j + 3]);
            s8x4_to_bf16x4(v.z, o[8 * j + 4], o[8 * j + 5]);
            s8x4_to_bf16x4(v.w, o[8 * j + 6], o[8 * j + 7]);
          }
        } else {
          // The box holds 128 k-rows of 128 P rows (byte r of k-row k in
          // chunk (r / 16) ^ (k % 8)).  Lane r reads the 32-bit word holding
          // its byte from four consecutive k-rows (lanes r, r ^ 1, r ^ 2,
          // r ^ 3 read the same word; the warp's 32 rows span two chunks, so
          // the reads are conflict-free) and gathers byte r % 4 of each into
          // one word of four consecutive k.
          const uint32_t box = sP + s * kPBytes;
          const uint32_t rc = (uint32_t)r >> 4, rw = (uint32_t)r & 12u;
          const uint32_t sel = ((uint32_t)r & 3u) | ((4u + ((uint32_t)r & 3u)) << 4);
#pragma unroll
          for (int kq = 0; kq < kKB / 4; ++kq) {
            uint32_t w4[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const uint32_t k = 4u * kq + i;
              w4[i] = ld_shared_u32(box + k * 128u + ((rc ^ (k & 7u)) << 4) + rw);
            }
            const uint32_t x = __byte_perm(__byte_perm(w4[0], w4[1], sel), __byte_perm(w4[2], w4[3], sel), 0x5410);
            s8x4_to_bf16x4(x, o[2 * kq], o[2 * kq + 1]);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(pempty_bar(s));  // this warp's rows of the P box are read
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
    griddep_wait();  // C (zeroed by the staging launch) is written below
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
      const int64_t q0 = (int64_t)w.tq * QN;
      if (p.add_into_c && p.c_tma) {  // the whole warp: rows past the matrix are clipped by the TMA
        reduce_rows_tma<QN>(&tmC, base + Cfg::kEpiOffset + (warp - 2) * 4096, lane, acc, p.swap != 0,
                            w.tp * kBM + quad * 32, (int32_t)q0, p.P_rows, p.Q_rows);
        continue;
      }
      const int64_t prow = (int64_t)w.tp * kBM + r;
      if (prow >= p.P_rows) continue;
      // partials (split-K of int16 / int8 outputs) have row pitch N; C has ldc
      const int64_t ld = (p.splits > 1 && p.out_bits != 32) ? (int64_t)p.N : p.ldc;
      if (p.swap)  // C[q][prow]: per element the warp's lanes store 32 consecutive columns
        store_row<QN>(p, acc, w.split, q0 * ld + prow, ld, q0);
      else         // C[prow][q]
        store_row<QN>(p, acc, w.split, prow * ld + q0, 1, q0);
    }
  }

  // the epilogue's TMA reductions have completed before the CTA leaves
  if (p.c_tma && warp >= 2 && warp < 2 + kEpiWarps && lane == 0) bulk_wait_all();
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

// Q's image for one (Q tile, k-block): QN rows x 128 K of bf16 as two
// 64-K halves of QN 128-byte rows, 16-byte chunk j of row r stored at chunk
// j ^ (r % 8) (the 128-byte swizzle).  One thread writes one 16-byte chunk
// (8 consecutive k of one row), reading Q(q, k) at src + q * sq + k * sk.
__global__ void __launch_bounds__(256)
    s8tm_stage_q_kernel(const int8_t *__restrict__ src, int64_t sq, int64_t sk, int Q_rows, int K, int qn,
                        int num_kb, uint4 *__restrict__ img, int64_t chunks, int32_t *__restrict__ zero_c,
                        int64_t c_rows, int64_t c_cols, int64_t ldc) {
  griddep_launch_dependents();  // the GEMM waits for completion before reading
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= chunks) {  // the remaining threads zero C (int32, the splits' sums are added into it)
    if (!zero_c) return;
    // four consecutive elements of a row per step, with one 16-byte store
    // when the row pitch and base allow it
    const bool vec = (reinterpret_cast<uintptr_t>(zero_c) & 15) == 0 && (ldc & 3) == 0;
    const int64_t quads = (c_cols + 3) >> 2, total = c_rows * quads;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x - chunks;
    for (int64_t e = t - chunks; e < total; e += stride) {
      const int64_t r = e / quads, c = (e - r * quads) << 2;
      int32_t *dst = zero_c + r * ldc + c;
      if (vec && c + 4 <= c_cols) {
        *reinterpret_cast<int4 *>(dst) = make_int4(0, 0, 0, 0);
      } else {
        for (int i = 0; i < 4 && c + i < c_cols; ++i) dst[i] = 0;
      }
    }
    return;
  }
  const int per_tile = 2 * qn * 8;  // 16-byte chunks per image
  const int64_t tile = t / per_tile;
  const int c = (int)(t - tile * per_tile);
  const int h = c / (qn * 8), rem = c - h * (qn * 8);
  const int row = rem >> 3, j = rem & 7;
  const int64_t tq = tile / num_kb, kb = tile - tq * num_kb;
  const int64_t q = tq * qn + row, k0 = kb * kKB + h * 64 + j * 8;
  uint32_t w[2] = {0u, 0u};
  if (q < Q_rows) {
    const int8_t *s = src + q * sq + k0 * sk;
    if (sk == 1 && k0 + 8 <= K && (reinterpret_cast<uintptr_t>(s) & 7) == 0) {
      const uint2 v = *reinterpret_cast<const uint2 *>(s);
      w[0] = v.x;
      w[1] = v.y;
    } else {
      for (int i = 0; i < 8; ++i)
        if (k0 + i < K) w[i >> 2] |= (uint32_t)(uint8_t)s[i * sk] << (8 * (i & 3));
    }
  }
  uint4 o;
  s8x4_to_bf16x4(w[0], o.x, o.y);
  s8x4_to_bf16x4(w[1], o.z, o.w);
  const int64_t at = tile * per_tile + h * (qn * 8) + row * 8 + (j ^ (row & 7));
  img[at] = o;
}

template <int QN, int SP, int SQ, int NA, bool PK>
cudaError_t launch_one(const CUtensorMap &tp, const CUtensorMap &tc, const S8tmParams &p, int grid,
                       cudaStream_t st) {
  using Cfg = S8tmCfg<QN, SP, SQ, NA>;
  auto kern = gemm_s8tm_kernel<QN, SP, SQ, NA, PK>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_ex(kern, dim3(grid), dim3(kThreadsS8tm), Cfg::kSmemBytes, st, 1, tp, tc, p);
}

}  // namespace

size_t s8tm_q_image_bytes(int qn, int64_t Q_rows, int64_t K) {
  const int64_t tiles_q = (Q_rows + qn - 1) / qn, num_kb = (K + kKB - 1) / kKB;
  return (size_t)tiles_q * num_kb * 2 * qn * 128;
}

cudaError_t launch_s8tm_stage_q(const int8_t *src, int64_t sq, int64_t sk, int64_t Q_rows, int64_t K, int qn,
                                void *img, int32_t *zero_c, int64_t c_rows, int64_t c_cols, int64_t ldc,
                                cudaStream_t st) {
  const int64_t num_kb = (K + kKB - 1) / kKB;
  const int64_t chunks = (int64_t)s8tm_q_image_bytes(qn, Q_rows, K) / 16;
  // more threads zero C when asked (up to 64K, a grid-stride loop over
  // four-element pieces of its rows)
  const int64_t quads = zero_c ? c_rows * ((c_cols + 3) / 4) : 0;
  const int64_t extra = quads < 65536 ? quads : 65536;
  if (chunks + extra == 0) return cudaSuccess;
  s8tm_stage_q_kernel<<<(unsigned)((chunks + extra + 255) / 256), 256, 0, st>>>(
      src, sq, sk, (int)Q_rows, (int)K, qn, (int)num_kb, static_cast<uint4 *>(img), chunks, zero_c, c_rows, c_cols,
      ldc);
  return cudaGetLastError();
}

cudaError_t launch_s8tm(int qn, bool p_kmajor, const CUtensorMap &tp, const CUtensorMap &tc, const S8tmParams &p,
                        int grid, cudaStream_t st) {
  // P stages x 16 KB + Q stages x (QN x 256 bytes): 9 x 16 + 2 x 32 KB
  // (QN 128) or 10 x 16 + 3 x 16 KB (QN 64), and four 4 KB epilogue blocks
  if (qn == 128)
    return p_kmajor ? launch_one<128, 9, 2, 4, true>(tp, tc, p, grid, st)
                    : launch_one<128, 9, 2, 4, false>(tp, tc, p, grid, st);
  return p_kmajor ? launch_one<64, 10, 3, 4, true>(tp, tc, p, grid, st)
                  : launch_one<64, 10, 3, 4, false>(tp, tc, p, grid, st);
}

}  // namespace gb300

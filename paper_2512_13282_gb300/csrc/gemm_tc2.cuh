// gemm_tc2.cuh -- the persistent tcgen05 GEMM on CTA pairs (cta_group::2).
//
// A cluster of two CTAs on neighbouring SMs owns a 256 x BN output tile.
// Each CTA loads its own 128 rows of A and one half (BN/2 rows/columns) of
// B into its shared memory; one thread of the leader CTA (rank 0) issues
// tcgen05.mma.cta_group::2 with M = 256, which reads the A and B halves of
// both CTAs and leaves rows 0..127 of the tile in the leader's TMEM and rows
// 128..255 in the peer's.  Per SM this halves the B bytes moved per flop,
// relieving L2 and shared-memory bandwidth, which is what limits the
// single-CTA kernel on large problems.
//
// Synchronisation (all waits bounded, see ptx.cuh):
//   full[s]   leader only: both CTAs' TMA loads of stage s complete on it;
//             the leader's producer posts the expected byte count of both.
//   empty[s]  both CTAs: the leader's MMA commit is multicast to both when
//             the MMAs reading stage s have finished.
//   accf[b]   both CTAs: multicast commit when accumulator b is complete.
//   acce[b]   leader only: all epilogue threads of both CTAs arrive (the
//             peer's remotely) when they have read accumulator b.
// Work units (tile, split) are walked per cluster; the int8 slab scheme and
// the epilogue are those of gemm_tc.cuh.
#pragma once
#include "gemm_tc.cuh"

namespace gb300 {

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// shared::cluster address of the same shared-memory offset in CTA `rank`.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t out;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(addr), "r"(rank));
  return out;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Arrive on an mbarrier given by its shared::cluster address (possibly in the
// peer CTA), with release semantics at cluster scope.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// TMA 2-D load into this CTA's shared memory whose completion is signalled
// on an mbarrier that may live in the peer CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void *tmap, int32_t c0, int32_t c1,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(bar_cluster)
      : "memory");
}

template <uint32_t kCols>
__device__ __forceinline__ void tmem_alloc_pair(uint32_t slot_smem) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot_smem), "n"(kCols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

template <uint32_t kCols>
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "n"(kCols) : "memory");
}

__device__ __forceinline__ void tc_mma_bf16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier at offset `bar` in both CTAs of the pair when
// the tcgen05 operations issued so far by this thread have completed.
__device__ __forceinline__ void tc_commit_pair_multicast(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          bar),
      "h"((uint16_t)0x3)
      : "memory");
}

template <int BN, int STAGES, bool B_KMAJOR, int EPI, int EPI_WARPS, int TMA_OUT>
struct Tc2Cfg {
  static constexpr int kHalfN = BN / 2;  // B extent (in N) each CTA loads
  static_assert(kHalfN % 16 == 0 && BN <= 256, "pair MMA N is a multiple of 32 up to 256");
  static_assert(B_KMAJOR || kHalfN % 64 == 0, "MN-major B halves are assembled from 64-wide boxes");
  static_assert(EPI_WARPS == 4 || EPI_WARPS == 8, "epilogue is one or two warpgroups");
  static constexpr uint32_t kBBytes = kHalfN * kRowBytes;
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;  // per CTA
  static constexpr uint32_t kTmemCols = pow2_at_least(2 * BN);
  static constexpr int kThreads = (2 + EPI_WARPS) * 32;
  static constexpr int kEpiThreads = EPI_WARPS * 32;
  static constexpr int kColsPerThread = BN / (EPI_WARPS / 4);
  static_assert(kColsPerThread % 16 == 0, "epilogue chunks are 32 columns, plus one of 16");
  static constexpr uint32_t kEpiWarpBytes = TMA_OUT == 1 ? 4096 : TMA_OUT == 2 ? 1024 : 0;  // one 32 x 32 block of 32-bit words
  static constexpr uint32_t kEpiOffset = STAGES * kStageBytes;
  static constexpr uint32_t kBarOffset = kEpiOffset + EPI_WARPS * kEpiWarpBytes;
  static constexpr uint32_t kNumBars = 2 * STAGES + 4 + 1;
  static constexpr uint32_t kSmemBytes = kBarOffset + kNumBars * 8 + 16 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA is 227 KB");
  static_assert(kSmemBytes == tc_smem_bytes(STAGES, kHalfN, EPI_WARPS, TMA_OUT), "layout and model agree");
  static_assert(kTmemCols <= 512, "TMEM has 512 columns");
};

// Launch with cluster dimensions (2,1,1) and an even grid; tiles_m counts
// 256-row tiles.
template <int BN, int STAGES, bool B_KMAJOR, int EPI, int EPI_WARPS, int TMA_OUT>
__global__ void __launch_bounds__(Tc2Cfg<BN, STAGES, B_KMAJOR, EPI, EPI_WARPS, TMA_OUT>::kThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmOut, const __grid_constant__ CUtensorMap tmWs,
                    const TcParams p) {
  using Cfg = Tc2Cfg<BN, STAGES, B_KMAJOR, EPI, EPI_WARPS, TMA_OUT>;
  const int out_tma = TMA_OUT != 0 ? p.out_tma : (int)kOutDirect;
  // the split tail's partials: through tmWs by the 4 KB staging blocks, or directly
  const int tail_out = (TMA_OUT == 1 && p.ws_tma) ? (int)kOutTmaWs : (int)kOutDirect;
  constexpr int kTileM = 2 * kBM;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *base_ptr = smem_raw + (base - raw);
  const uint32_t sA = base;
  const uint32_t sB = base + STAGES * kABytes;
  const uint32_t bars = base + Cfg::kBarOffset;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(base_ptr + Cfg::kBarOffset + Cfg::kNumBars * 8);
  volatile uint32_t *abort_flag = tmem_slot + 1;

  auto full_bar = [&](uint32_t s) { return bars + 8u * s; };
  auto empty_bar = [&](uint32_t s) { return bars + 8u * (STAGES + s); };
  auto accf_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + b); };
  auto acce_bar = [&](uint32_t b) { return bars + 8u * (2 * STAGES + 2 + b); };
  const uint32_t drain_bar = bars + 8u * (2 * STAGES + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cluster = blockIdx.x >> 1;
  const int num_clusters = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), 2 * Cfg::kEpiThreads);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (out_tma != kOutDirect) tma_prefetch_desc(&tmOut);
    if (p.tail_splits > 0 && tail_out != kOutDirect) tma_prefetch_desc(&tmWs);
  }
  __syncwarp();
  if (warp == 1) tmem_alloc_pair<Cfg::kTmemCols>(smem_addr(tmem_slot));
  tc_fence_before_sync();
  cluster_sync_all();  // barriers of both CTAs initialised, TMEM allocated
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  // Everything above only touched this CTA's shared memory, TMEM and the
  // kernel parameters, and may overlap the previous kernel of the stream;
  // global memory is touched only after that kernel has completed.
  griddep_wait();

  const int num_units = tc_num_units(p);
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

  if (warp == 0) {
    // ---------------------------------------------- TMA producer (both CTAs)
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int u = cluster; ok && u < num_units; u += num_clusters) {
        const Unit w = decode_unit(p, u);
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          const uint32_t s = g % STAGES, ph = (g / STAGES) & 1u;
          if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, p.err, p.wait_limit_ns)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full_bar(s), 2 * Cfg::kStageBytes);
          const uint32_t fb = mapa_shared(full_bar(s), 0);
          tma_load_2d_pair(sA + s * kABytes, &tmA, kb * kBK, w.tm * kTileM + (int)rank * kBM, fb);
          const uint32_t b_dst = sB + s * Cfg::kBBytes;
          const int n0 = w.tn * BN + (int)rank * Cfg::kHalfN;
          if constexpr (B_KMAJOR) {
            tma_load_2d_pair(b_dst, &tmB, kb * kBK, n0, fb);
          } else {
#pragma unroll
            for (int j = 0; j < Cfg::kHalfN / 64; ++j)
              tma_load_2d_pair(b_dst + j * (kBK * 128), &tmB, n0 + 64 * j, kb * kBK, fb);
          }
          ++g;
        }
      }
      if (leader) {
        const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
        for (uint32_t i = first; i < g; ++i)
          mbar_wait_drain(full_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
      } else {
        // the peer's loads complete on the leader's barriers; wait until the
        // leader's MMAs have released the stages they filled
        const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
        for (uint32_t i = first; i < g; ++i)
          mbar_wait_drain(empty_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && leader) {
      constexpr uint32_t idesc = idesc_bf16_f32(kTileM, BN, !B_KMAJOR);
      uint32_t g = 0, acc_cnt = 0;
      bool ok = true;
      for (int u = cluster; ok && u < num_units; u += num_clusters) {
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
            if (!mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t a0 = sA + s * kABytes;
            const uint32_t b0 = sB + s * Cfg::kBBytes;
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              const uint64_t ad = smem_desc_sw128(a0 + k * 32, 16, 1024);
              const uint64_t bd = B_KMAJOR ? smem_desc_sw128(b0 + k * 32, 16, 1024)
                                           : smem_desc_sw128(b0 + k * 2048, kBK * 128, 1024);
              tc_mma_bf16_pair(d_tmem, ad, bd, idesc, (kb > kb_s || k > 0) ? 1u : 0u);
            }
            tc_commit_pair_multicast(empty_bar(s));
            ++g;
          }
          if (!ok) break;
          tc_commit_pair_multicast(accf_bar(b));
          ++acc_cnt;
        }
      }
      tc_commit_pair_multicast(drain_bar);
      mbar_wait_drain(drain_bar, 0, kDrainNs);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ epilogue (both CTAs)
    constexpr int CPT = Cfg::kColsPerThread;
    const int ew = warp - 2;
    const int quad = warp & 3;
    const int colpart = ew >> 2;
    const int row_in_tile = (int)rank * kBM + quad * 32 + lane;
    const bool ws_vec = (p.N & 3) == 0;
    const uint32_t ebuf = base + Cfg::kEpiOffset + ew * Cfg::kEpiWarpBytes;
    uint32_t acc_cnt = 0;
    bool ok = true;
    for (int u = cluster; ok && u < num_units; u += num_clusters) {
      const Unit w = decode_unit(p, u);
      const bool split = w.part != 0;                  // partials of this unit, not C
      const bool tail = split && p.tail_splits > 0;    // ... of a split-tail tile
      const int uo = tail ? tail_out : out_tma;
      const CUtensorMap *om = tail ? &tmWs : &tmOut;
      // partial coordinates: a split-tail tile's partials are a compact
      // block (origin px, py of the matrix; rows of pn words), split-K
      // partials whole planes of C's shape
      const int px = tail ? w.tn * BN : 0;
      const int py = tail ? (w.tm - w.slot) * kTileM : 0;
      const int pn = tail ? BN : p.N;
      const int64_t pm = tail ? (int64_t)(p.tiles_m * p.tiles_n - p.tail_first) * kTileM : (int64_t)p.M;
      const int64_t row = (int64_t)w.tm * kTileM + row_in_tile;
      const bool row_ok = row < p.M;
      const int col0 = w.tn * BN + colpart * CPT;
      const int y0 = w.tm * kTileM + (int)rank * kBM + quad * 32;  // first row of this warp's blocks
      if constexpr (EPI == kEpiS32) {
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
            tmem_ld<32>(t0 + c * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) acc[c * 32 + i] += __float2int_rn(__uint_as_float(r[i]));
          }
          if constexpr (CPT % 32 != 0) {
            constexpr int kTail = (CPT / 32) * 32;
            uint32_t r[16];
            tmem_ld<16>(t0 + kTail, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[kTail + i] += __float2int_rn(__uint_as_float(r[i]));
          }
          tc_fence_before_sync();
          mbar_arrive_cluster(mapa_shared(acce_bar(b), 0));
          ++acc_cnt;
        }
        if (!ok) break;
        // split-K partials stay int32; the reduction requantises
        uint32_t *wrow = split ? reinterpret_cast<uint32_t *>(p.ws) + ((int64_t)w.split * pm + (row - py)) * pn
                               : nullptr;
        if (uo != kOutDirect) {
#pragma unroll
          for (int c = 0; c < CPT / 32; ++c) {
            uint32_t v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = static_cast<uint32_t>(acc[c * 32 + i]);
            const int x = col0 + c * 32;
            if (uo == kOutTmaWs)
              tma_out_words32<true>(om, ebuf, lane, v, x - px, y0 - py, w.split, y0 < p.M && x < p.N);
            else if (p.out_bits == 32)
              tma_out_words32<false>(om, ebuf, lane, v, x, y0, 0, y0 < p.M && x < p.N);
            else
              tma_out_narrow(om, ebuf, lane, v, p.out_bits, p.out_shift, x, y0, y0 < p.M && x < p.N);
          }
          if constexpr (CPT % 32 != 0) {  // a 16-column tail: each lane stores its row
            constexpr int kTail = (CPT / 32) * 32;
            if (row_ok) {
              uint32_t v[16];
#pragma unroll
              for (int i = 0; i < 16; ++i) v[i] = static_cast<uint32_t>(acc[kTail + i]);
              if (split)
                store_words<16>(wrow, col0 + kTail - px, pn, ws_vec, v);
              else
                store_s8_result<16>(p, row, col0 + kTail, v);
            }
          }
        } else if (row_ok) {
#pragma unroll
          for (int c = 0; c < CPT / 32; ++c) {
            uint32_t v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = static_cast<uint32_t>(acc[c * 32 + i]);
            if (split)
              store_words<32>(wrow, col0 + c * 32 - px, pn, ws_vec, v);
            else
              store_s8_result<32>(p, row, col0 + c * 32, v);
          }
          if constexpr (CPT % 32 != 0) {
            constexpr int kTail = (CPT / 32) * 32;
            uint32_t v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = static_cast<uint32_t>(acc[kTail + i]);
            if (split)
              store_words<16>(wrow, col0 + kTail - px, pn, ws_vec, v);
            else
              store_s8_result<16>(p, row, col0 + kTail, v);
          }
        }
      } else {
        const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait(accf_bar(b), aph, abort_flag, p.err, p.wait_limit_ns))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t t0 = tmem_base + b * BN + ((uint32_t)(quad * 32) << 16) + colpart * CPT;
        uint16_t *crow = reinterpret_cast<uint16_t *>(p.C) + row * p.ldc;
        uint32_t *wrow = split ? reinterpret_cast<uint32_t *>(p.ws) + ((int64_t)w.split * pm + (row - py)) * pn
                               : nullptr;
#pragma unroll 1
        for (int c = 0; c < CPT / 32; ++c) {
          uint32_t r[32];
          tmem_ld<32>(t0 + c * 32, r);
          tmem_ld_wait();
          const int x = col0 + c * 32;
          if (TMA_OUT == 1 && uo == kOutTmaWs) {
            tma_out_words32<true>(om, ebuf, lane, r, x - px, y0 - py, w.split, y0 < p.M && x < p.N);
          } else if (TMA_OUT == 1 && uo == kOutTmaC) {
            tma_out_bf16x32(om, ebuf, lane, r, x, y0, y0 < p.M && x < p.N);
          } else if (TMA_OUT == 2 && uo == kOutTmaC) {
            tma_out_bf16x16x2(om, ebuf, lane, r, x, y0, p.M, p.N);
          } else if (row_ok) {
            if (split)
              store_words<32>(wrow, x - px, pn, ws_vec, r);
            else
              store_bf16<32>(crow, x, p.N, p.c_vec != 0, r);
          }
        }
        if constexpr (CPT % 32 != 0) {
          constexpr int kTail = (CPT / 32) * 32;
          uint32_t r[16];
          tmem_ld<16>(t0 + kTail, r);
          tmem_ld_wait();
          if (row_ok) {
            if (split)
              store_words<16>(wrow, col0 + kTail - px, pn, ws_vec, r);
            else
              store_bf16<16>(crow, col0 + kTail, p.N, p.c_vec != 0, r);
          }
        }
        tc_fence_before_sync();
        mbar_arrive_cluster(mapa_shared(acce_bar(b), 0));
        ++acc_cnt;
      }
    }
  }

  if (TMA_OUT && warp >= 2 && lane == 0) bulk_wait_all();  // this warp's TMA stores have landed
  griddep_launch_dependents();  // e.g. the split-K reduction may start setting up
  __syncwarp();
  tc_fence_before_sync();
  cluster_sync_all();  // no remote arrival or load may target a CTA that has left
  if (warp == 1) {
    __syncwarp();
    tc_fence_after_sync();
    tmem_dealloc_pair<Cfg::kTmemCols>(tmem_base);
  }
}

}  // namespace gb300

// gemm_tc.cuh -- persistent, warp-specialised tcgen05 GEMM kernel.
//
// One CTA per SM loops over output tiles (the paper's output-stationary
// mapping, Sec. 4.2.1: M and N are spread in space over independent workers,
// K is reduced in time into a stationary accumulator).  Roles:
//   warp 0 (one lane)  TMA producer: streams 128 x 64 A boxes and BN x 64 B
//                      boxes into a STAGES-deep shared-memory ring (the
//                      paper's double-buffered L1/L2 input tiles, Sec. 4.2.1,
//                      deepened), each stage guarded by a full/empty mbarrier
//                      pair.  The box shapes and the 128-byte swizzle play the
//                      part of the paper's on-the-fly DMA layout transforms
//                      (Sec. 4.3): matrices stay row-/column-major in memory.
//   warp 1 (one lane)  MMA issuer: tcgen05.mma kind::f16 (bf16 x bf16 -> fp32)
//                      into one of two TMEM accumulators; the first MMA of a
//                      tile overwrites instead of accumulating, which takes
//                      the place of the paper's zeroing kernel (Sec. 4.2.1).
//   warps 2..          epilogue: TMEM -> registers -> bf16 (RNE), int32, or
//                      int32 requantised to int16 / int8 -> a 32-row block
//                      in the warp's own shared memory (swizzled as the TMA
//                      expects) -> one TMA tensor store per block, which
//                      writes whole lines of C and clips at the M/N edges.
//                      Stores that each lane makes to its own row touch 32
//                      lines per instruction and compete with the operand
//                      traffic; lanes store their rows directly only where
//                      C's address or pitch rules TMA out, and in the int8
//                      variants that trade the staging blocks for a pipeline
//                      stage (long reductions).  Two accumulators let the
//                      epilogue of one tile overlap the main loop of the
//                      next (the paper keeps a single C buffer for lack of
//                      L1 space, Sec. 5.3.2; TMEM has room for two).
//
// Exact int8 emulation (kEpiS32): int8 operands, staged as bf16 (every int8
// value is exact in bf16), are multiplied on the bf16 pipe.  A product is at
// most 2^14 in magnitude, so any partial sum of at most 1024 of them is an
// integer of magnitude <= 2^24 and exact in fp32.  The MMA warp therefore
// closes the accumulator every `slab_kb` k-blocks (slab_kb * 64 <= 1024 K
// elements); the epilogue converts each slab's fp32 sums to int32 (exactly)
// and adds them in int32 registers.  The final int32 is exact whenever the
// true result fits int32.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstdint>

#include "ptx.cuh"

namespace gb300 {

constexpr int kBM = 128;                    // MMA M (rows of C per tile)
constexpr int kBK = 64;                     // K per stage: 64 bf16 = 128 bytes
constexpr uint32_t kRowBytes = kBK * 2;     // one 128-byte swizzle row
constexpr uint32_t kABytes = kBM * kRowBytes;

enum EpiKind : int { kEpiBf16 = 0, kEpiS32 = 1 };

struct TcParams {
  int M, N, K;
  int tiles_m, tiles_n;
  int num_kb;        // ceil(K / kBK)
  int splits;        // split-K factor (1: none)
  int kb_per_split;  // k-blocks per split
  int slab_kb;       // k-blocks per accumulator slab (>= kb_per_split for bf16)
  int group_m;       // tiles of M per rasterisation group
  void *C;           // bf16 or int32 output, row-major, leading dimension ldc
  int64_t ldc;
  int c_vec;         // C rows 16-byte aligned (informational; stores check each address)
  void *ws;          // partials (fp32 or int32): split-K, splits x M x N words; a split tail, compact (below)
  uint32_t *err;     // device error word
  uint64_t wait_limit_ns;
  int out_bits;      // int8 path: 32 (exact int32 C), 16 or 8 (requantised C)
  int out_shift;     // int8 path with out_bits < 32: right shift, 0..31
  int out_tma;       // kOutDirect, kOutTmaC (tmOut maps C) or kOutTmaWs (tmOut maps the partials)
  // Split tail (tail_splits >= 2, splits == 1): the tiles of the last,
  // partly filled round -- raster positions tail_first .. -- are each split
  // into tail_splits units of tail_kb_per k-blocks that write partials for
  // the reduction kernel, so that the round takes 1 / tail_splits of a
  // tile's time; every other tile is one unit writing C.  tail_first is a
  // whole number of rounds of units.  The tail's partials are compact:
  // plane s holds, for the tail tile at raster position tail_first + i, a
  // block of tile rows x BN 32-bit words at row i * tile rows (row pitch BN).
  // ws_tma: they are stored through tmWs (else directly).
  int tail_first, tail_splits, tail_kb_per, ws_tma;
};

// How the epilogue writes its results.
enum OutMode : int { kOutDirect = 0, kOutTmaC = 1, kOutTmaWs = 2 };

__host__ __device__ constexpr uint32_t pow2_at_least(uint32_t x) {
  uint32_t p = 32;
  while (p < x) p <<= 1;
  return p;
}

// Shared memory of a tensor-core kernel (the memory constraint of the
// paper's tile model, Sec. 4.5.1 Eq. 5, on one SM): STAGES operand stages
// (a 128 x 64 bf16 A box and a bn_cta x 64 B box), the epilogue warps'
// output staging blocks (4 KB, 1 KB or none each), two barriers per stage
// and five more, the TMEM address and abort words, and the slack that
// aligns the ring to 1024 bytes.
__host__ __device__ constexpr uint32_t tc_smem_bytes(int stages, int bn_cta, int epi_warps, int tma_out) {
  return (uint32_t)stages * (kABytes + (uint32_t)bn_cta * kRowBytes) +
         (uint32_t)epi_warps * (tma_out == 1 ? 4096u : tma_out == 2 ? 1024u : 0u) +
         (uint32_t)(2 * stages + 5) * 8u + 16u + 1024u;
}

// The deepest pipeline that fits the 227 KB a CTA may use: every compiled
// kernel takes this many stages.
__host__ __device__ constexpr int tc_max_stages(int bn_cta, int epi_warps, int tma_out) {
  int s = 1;
  while (tc_smem_bytes(s + 1, bn_cta, epi_warps, tma_out) <= 232448u) ++s;
  return s;
}

template <int BN, int STAGES, bool B_KMAJOR, int EPI, int EPI_WARPS, int TMA_OUT>
struct TcCfg {
  // MMA N for M = 128 is a multiple of 16 up to 256; the epilogue moves 32
  // columns per TMEM load; an MN-major B tile is assembled from 64-wide boxes.
  static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "BN must be 64..256, a multiple of 32");
  static_assert(B_KMAJOR || BN % 64 == 0, "MN-major B needs BN a multiple of 64");
  static_assert(EPI_WARPS == 4 || EPI_WARPS == 8, "epilogue is one or two warpgroups");
  static constexpr uint32_t kBBytes = BN * kRowBytes;
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kTmemCols = pow2_at_least(2 * BN);  // two fp32 accumulators
  static constexpr int kThreads = (2 + EPI_WARPS) * 32;
  static constexpr int kColsPerThread = BN / (EPI_WARPS / 4);
  static_assert(kColsPerThread % 16 == 0, "epilogue chunks are 32 columns, plus one of 16");
  // TMA_OUT 1: per epilogue warp, one 32 x 32 block of 32-bit words (int32
  // results or split-K partials of either path; bf16 results use half of
  // it); TMA_OUT 2 (bf16 C only): a 1 KB block of 32 rows x 16 bf16
  static constexpr uint32_t kEpiWarpBytes = TMA_OUT == 1 ? 4096 : TMA_OUT == 2 ? 1024 : 0;
  static constexpr uint32_t kEpiOffset = STAGES * kStageBytes;  // 1024-byte aligned
  static constexpr uint32_t kBarOffset = kEpiOffset + EPI_WARPS * kEpiWarpBytes;
  static constexpr uint32_t kNumBars = 2 * STAGES + 4 + 1;
  static constexpr uint32_t kSmemBytes = kBarOffset + kNumBars * 8 + 16 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA is 227 KB");
  static_assert(kSmemBytes == tc_smem_bytes(STAGES, BN, EPI_WARPS, TMA_OUT), "layout and model agree");
  static_assert(kTmemCols <= 512, "TMEM has 512 columns");
};

struct Unit {
  int tm, tn, split, kb0, kb1;
  int part;  // 1: the unit writes split-K partials (plane `split`), 0: C
  int slot;  // split-tail units: the tile's place among the tail tiles
};

// Raster position t -> output tile (tm, tn).  Tiles are visited in groups of
// group_m M-tiles so that CTAs running at the same time share A rows and B
// columns in L2.  The split-K reduction of a split tail walks the same
// positions.
__host__ __device__ __forceinline__ void raster_tile(int t, int tiles_m, int tiles_n, int group_m, int *tm,
                                                     int *tn) {
  const int group = group_m * tiles_n;
  const int gid = t / group;
  const int first_m = gid * group_m;
  const int gm = tiles_m - first_m < group_m ? tiles_m - first_m : group_m;
  const int local = t - gid * group;
  *tm = first_m + local % gm;
  *tn = local / gm;
}

// Work units of a launch: tiles x splits, or the whole tiles before the
// split tail plus tail_splits units per tail tile.
__device__ __forceinline__ int tc_num_units(const TcParams &p) {
  const int num_tiles = p.tiles_m * p.tiles_n;
  return p.tail_splits > 0 ? p.tail_first + (num_tiles - p.tail_first) * p.tail_splits : num_tiles * p.splits;
}

// Work unit u -> (tile, split, k-blocks).  With split-K, unit u is split
// u / tiles of raster position u % tiles; with a split tail, units below
// tail_first are whole tiles and the rest split the tail tiles.
__device__ __forceinline__ Unit decode_unit(const TcParams &p, int u) {
  const int num_tiles = p.tiles_m * p.tiles_n;
  Unit w;
  int t;
  if (p.tail_splits > 0 && u >= p.tail_first) {
    const int tail = num_tiles - p.tail_first;
    const int v = u - p.tail_first;
    w.split = v / tail;
    t = p.tail_first + (v - w.split * tail);
    w.kb0 = w.split * p.tail_kb_per;
    w.kb1 = min(p.num_kb, w.kb0 + p.tail_kb_per);
    w.part = 1;
    w.slot = t - p.tail_first;
  } else {
    w.slot = 0;
    w.split = u / num_tiles;
    t = u - w.split * num_tiles;
    w.kb0 = w.split * p.kb_per_split;
    w.kb1 = min(p.num_kb, w.kb0 + p.kb_per_split);
    w.part = p.splits > 1 ? 1 : 0;
  }
  raster_tile(t, p.tiles_m, p.tiles_n, p.group_m, &w.tm, &w.tn);
  return w;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // round to nearest even
  return *reinterpret_cast<uint32_t *>(&v);
}

// Reduced-precision int8 outputs (Sec. 5.1 reduces int8 GEMM outputs to 16
// and 8 bits): the exact sum divided by 2^shift, rounded to nearest with
// ties to even, saturated to the output type.  RneShift does the division
// and rounding in 32-bit arithmetic: q0 = a >> shift is the floor, r the
// non-negative remainder a mod 2^shift, and (r + (q0 odd) + 2^(shift-1) - 1)
// >> shift is 1 exactly when r > 2^(shift-1), or r = 2^(shift-1) with q0
// odd; that sum stays below 2^32 for every shift 0..31.  With shift 0 all
// terms but q0 vanish.
struct RneShift {
  int shift;
  uint32_t mask, odd, half_m1;
  __host__ __device__ explicit RneShift(int s)
      : shift(s), mask(s ? (1u << s) - 1u : 0u), odd(s ? 1u : 0u), half_m1(s ? (1u << (s - 1)) - 1u : 0u) {}
  __host__ __device__ __forceinline__ int32_t operator()(int32_t a) const {
    const int32_t q0 = a >> shift;
    const uint32_t t = (static_cast<uint32_t>(a) & mask) + (static_cast<uint32_t>(q0) & odd) + half_m1;
    return q0 + static_cast<int32_t>(t >> shift);
  }
};

// The same, saturated to [lo, hi].
__host__ __device__ __forceinline__ int32_t requantize_s32(int32_t a, int shift, int32_t lo, int32_t hi) {
  const int32_t q = RneShift(shift)(a);
  return q < lo ? lo : (q > hi ? hi : q);
}

// Store `bytes` (a multiple of 16) of a row chunk that lies fully inside
// the matrix, with the widest stores the chunk's start address allows
// (16, 8 or 4 bytes): rows of a C whose leading dimension is not a multiple
// of 16 bytes are still stored without falling back to one store per
// element.  `w` holds the chunk as 32-bit words.
template <int NWORDS>
__device__ __forceinline__ void store_chunk_aligned(void *dst, const uint32_t (&w)[NWORDS]) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(dst);
  if ((a & 15) == 0) {
    uint4 *d = reinterpret_cast<uint4 *>(dst);
#pragma unroll
    for (int i = 0; i < NWORDS / 4; ++i) d[i] = make_uint4(w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
  } else if ((a & 7) == 0) {
    uint2 *d = reinterpret_cast<uint2 *>(dst);
#pragma unroll
    for (int i = 0; i < NWORDS / 2; ++i) d[i] = make_uint2(w[2 * i], w[2 * i + 1]);
  } else {
    uint32_t *d = reinterpret_cast<uint32_t *>(dst);
#pragma unroll
    for (int i = 0; i < NWORDS; ++i) d[i] = w[i];
  }
}

// Store W (16 or 32) consecutive 32-bit words of one row (fp32 partials or
// int32); element-wise only where the chunk crosses column N.
template <int W>
__device__ __forceinline__ void store_words(uint32_t *dst, int col, int N, bool vec, const uint32_t (&v)[W]) {
  (void)vec;
  if (col + W <= N) {
    store_chunk_aligned<W>(dst + col, v);
  } else {
#pragma unroll
    for (int i = 0; i < W; ++i)
      if (col + i < N) dst[col + i] = v[i];
  }
}

// Round W fp32 accumulator words to bf16 (nearest even) and store them.
template <int W>
__device__ __forceinline__ void store_bf16(uint16_t *dst, int col, int N, bool vec, const uint32_t (&r)[W]) {
  (void)vec;
  uint32_t h[W / 2];
#pragma unroll
  for (int i = 0; i < W / 2; ++i) h[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
  if (col + W <= N && (reinterpret_cast<uintptr_t>(dst + col) & 3) == 0) {
    store_chunk_aligned<W / 2>(dst + col, h);
  } else {
#pragma unroll
    for (int i = 0; i < W; ++i)
      if (col + i < N) dst[col + i] = static_cast<uint16_t>(h[i >> 1] >> (16 * (i & 1)));
  }
}

// Store W (16 or 32) int32 results of row `row`, columns [col, col + W)
// clipped at N, into C: as int32, or requantised to int16 / int8 and packed
// into 32-bit words (per element where the chunk crosses N or the address
// is not 4-byte aligned).
template <int W>
__device__ __forceinline__ void store_s8_result(const TcParams &p, int64_t row, int col, const uint32_t (&v)[W]) {
  if (p.out_bits == 32) {
    store_words<W>(reinterpret_cast<uint32_t *>(p.C) + row * p.ldc, col, p.N, true, v);
    return;
  }
  const int32_t hi = (1 << (p.out_bits - 1)) - 1, lo = -hi - 1;
  int32_t q[W];
#pragma unroll
  for (int i = 0; i < W; ++i) q[i] = requantize_s32(static_cast<int32_t>(v[i]), p.out_shift, lo, hi);
  const bool full = col + W <= p.N;
  if (p.out_bits == 16) {
    int16_t *dst = reinterpret_cast<int16_t *>(p.C) + row * p.ldc + col;
    if (full && (reinterpret_cast<uintptr_t>(dst) & 3) == 0) {
      uint32_t h[W / 2];
#pragma unroll
      for (int i = 0; i < W / 2; ++i)
        h[i] = (static_cast<uint32_t>(q[2 * i]) & 0xFFFFu) | (static_cast<uint32_t>(q[2 * i + 1]) << 16);
      store_chunk_aligned<W / 2>(dst, h);
    } else {
#pragma unroll
      for (int i = 0; i < W; ++i)
        if (col + i < p.N) dst[i] = static_cast<int16_t>(q[i]);
    }
  } else {
    int8_t *dst = reinterpret_cast<int8_t *>(p.C) + row * p.ldc + col;
    if (full && (reinterpret_cast<uintptr_t>(dst) & 3) == 0) {
      uint32_t h[W / 4];
#pragma unroll
      for (int i = 0; i < W / 4; ++i)
        h[i] = (static_cast<uint32_t>(q[4 * i]) & 0xFFu) | ((static_cast<uint32_t>(q[4 * i + 1]) & 0xFFu) << 8) |
               ((static_cast<uint32_t>(q[4 * i + 2]) & 0xFFu) << 16) | (static_cast<uint32_t>(q[4 * i + 3]) << 24);
      store_chunk_aligned<W / 4>(dst, h);
    } else {
#pragma unroll
      for (int i = 0; i < W; ++i)
        if (col + i < p.N) dst[i] = static_cast<int8_t>(q[i]);
    }
  }
}

// TMA-store epilogue.  A warp stages 32 rows (lane = row) x 32 columns in
// its shared-memory block laid out as the tensor map's swizzle expects, then
// lane 0 stores the block with one TMA tensor store.  The block is reused
// once the previous store has read it.  `in_range`: the block's first row
// and column lie inside the output (the TMA clips the rest).
//
// 32-bit words (int32 results, fp32/int32 split-K partials): 128-byte rows,
// 128-byte swizzle (16-byte chunk j of row r lands at chunk j ^ (r % 8)).
template <bool WS>
__device__ __forceinline__ void tma_out_words32(const CUtensorMap *tm, uint32_t buf, int lane,
                                                const uint32_t (&v)[32], int x, int y, int z, bool in_range) {
  if (lane == 0) bulk_wait_read_all();
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 8; ++j)
    st_shared_v4(buf + lane * 128 + ((j ^ (lane & 7)) << 4), v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0 && in_range) {
    if constexpr (WS)
      tma_store_3d(tm, buf, x, y, z);
    else
      tma_store_2d(tm, buf, x, y);
    bulk_commit();
  }
}

// bf16 results: 32 fp32 accumulator words rounded to 32 bf16 (64-byte rows),
// 64-byte swizzle (chunk j of row r lands at chunk j ^ ((r / 2) % 4)).
__device__ __forceinline__ void tma_out_bf16x32(const CUtensorMap *tm, uint32_t buf, int lane, const uint32_t (&r)[32],
                                                int x, int y, bool in_range) {
  uint32_t h[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) h[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
  if (lane == 0) bulk_wait_read_all();
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 4; ++j)
    st_shared_v4(buf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4), h[4 * j], h[4 * j + 1], h[4 * j + 2], h[4 * j + 3]);
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0 && in_range) {
    tma_store_2d(tm, buf, x, y);
    bulk_commit();
  }
}

// bf16 results through a 1 KB block: the 32 columns go out as two 16-column
// halves (32-byte rows, 32-byte swizzle: chunk j of row r lands at chunk
// j ^ ((r / 4) % 2)), one after the other.
__device__ __forceinline__ void tma_out_bf16x16x2(const CUtensorMap *tm, uint32_t buf, int lane,
                                                  const uint32_t (&r)[32], int x, int y, int M, int N) {
  uint32_t h[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) h[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
  const uint32_t sw = (lane >> 2) & 1;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    if (lane == 0) bulk_wait_read_all();
    __syncwarp();
    st_shared_v4(buf + lane * 32 + ((0u ^ sw) << 4), h[8 * half], h[8 * half + 1], h[8 * half + 2], h[8 * half + 3]);
    st_shared_v4(buf + lane * 32 + ((1u ^ sw) << 4), h[8 * half + 4], h[8 * half + 5], h[8 * half + 6],
                 h[8 * half + 7]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0 && y < M && x + 16 * half < N) {
      tma_store_2d(tm, buf, x + 16 * half, y);
      bulk_commit();
    }
  }
}

// Requantised int8-path results (int16 or int8 C): 32 int32 sums of a row
// requantised and packed into 64-byte (int16; 64-byte swizzle) or 32-byte
// (int8; 32-byte swizzle: chunk j of row r lands at chunk j ^ ((r / 4) % 2))
// rows, then stored like the other blocks.
__device__ __forceinline__ void tma_out_narrow(const CUtensorMap *tm, uint32_t buf, int lane, const uint32_t (&v)[32],
                                               int bits, int shift, int x, int y, bool in_range) {
  // rounding in 32-bit arithmetic, saturation and packing by cvt.pack.sat
  const RneShift rq(shift);
  uint32_t h[16];
  if (bits == 16) {
#pragma unroll
    for (int i = 0; i < 16; ++i) h[i] = pack_sat_s16x2(rq((int32_t)v[2 * i]), rq((int32_t)v[2 * i + 1]));
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i)
      h[i] = pack_sat_s8x4(rq((int32_t)v[4 * i]), rq((int32_t)v[4 * i + 1]), rq((int32_t)v[4 * i + 2]),
                           rq((int32_t)v[4 * i + 3]));
  }
  if (lane == 0) bulk_wait_read_all();
  __syncwarp();
  if (bits == 16) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      st_shared_v4(buf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4), h[4 * j], h[4 * j + 1], h[4 * j + 2],
                   h[4 * j + 3]);
  } else {
#pragma unroll
    for (int j = 0; j < 2; ++j)
      st_shared_v4(buf + lane * 32 + ((j ^ ((lane >> 2) & 1)) << 4), h[4 * j], h[4 * j + 1], h[4 * j + 2],
                   h[4 * j + 3]);
  }
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0 && in_range) {
    tma_store_2d(tm, buf, x, y);
    bulk_commit();
  }
}

// One 32-column chunk of a lane's int32 sums (row `row`, columns x ..): to
// C (int32, or requantised) or to the split's partials (wrow), through the
// warp's TMA staging block when out_tma says so (the warp's rows y0 ..),
// else directly.
__device__ __forceinline__ void store_s32_chunk(const TcParams &p, const CUtensorMap *tm, uint32_t ebuf, int lane,
                                                int out_tma, const uint32_t (&v)[32], int x, int y0, int split,
                                                bool row_ok, int64_t row, uint32_t *wrow, bool ws_vec, int px,
                                                int py, int pn) {
  if (out_tma != kOutDirect) {
    if (out_tma == kOutTmaWs)
      tma_out_words32<true>(tm, ebuf, lane, v, x - px, y0 - py, split, y0 < p.M && x < p.N);
    else if (p.out_bits == 32)
      tma_out_words32<false>(tm, ebuf, lane, v, x, y0, 0, y0 < p.M && x < p.N);
    else
      tma_out_narrow(tm, ebuf, lane, v, p.out_bits, p.out_shift, x, y0, y0 < p.M && x < p.N);
  } else if (row_ok) {
    if (wrow)
      store_words<32>(wrow, x - px, pn, ws_vec, v);
    else
      store_s8_result<32>(p, row, x, v);
  }
}

template <int W>
__device__ __forceinline__ void tmem_ld(uint32_t taddr, uint32_t (&r)[W]) {
  if constexpr (W == 32)
    tmem_ld_32x32b_x32(taddr, r);
  else
    tmem_ld_32x32b_x16(taddr, r);
}

template <int BN, int STAGES, bool B_KMAJOR, int EPI, int EPI_WARPS, int TMA_OUT>
__global__ void __launch_bounds__(TcCfg<BN, STAGES, B_KMAJOR, EPI, EPI_WARPS, TMA_OUT>::kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmOut, const __grid_constant__ CUtensorMap tmWs,
                   const TcParams p) {
  using Cfg = TcCfg<BN, STAGES, B_KMAJOR, EPI, EPI_WARPS, TMA_OUT>;
  const int out_tma = TMA_OUT != 0 ? p.out_tma : (int)kOutDirect;
  // the split tail's partials: through tmWs by the 4 KB staging blocks, or directly
  const int tail_out = (TMA_OUT == 1 && p.ws_tma) ? (int)kOutTmaWs : (int)kOutDirect;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-byte alignment
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

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), EPI_WARPS * 32);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (out_tma != kOutDirect) tma_prefetch_desc(&tmOut);
    if (p.tail_splits > 0 && tail_out != kOutDirect) tma_prefetch_desc(&tmWs);
  }
  if (warp == 1) tmem_alloc<Cfg::kTmemCols>(smem_addr(tmem_slot));
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *tmem_slot;
  // Everything above only touched this CTA's shared memory, TMEM and the
  // kernel parameters, and may overlap the previous kernel of the stream;
  // global memory is touched only after that kernel has completed.
  griddep_wait();

  const int num_units = tc_num_units(p);
  constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

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
          mbar_arrive_expect_tx(full_bar(s), Cfg::kStageBytes);
          tma_load_2d(sA + s * kABytes, &tmA, kb * kBK, w.tm * kBM, full_bar(s));
          const uint32_t b_dst = sB + s * Cfg::kBBytes;
          if constexpr (B_KMAJOR) {
            tma_load_2d(b_dst, &tmB, kb * kBK, w.tn * BN, full_bar(s));
          } else {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tma_load_2d(b_dst + j * (kBK * 128), &tmB, w.tn * BN + 64 * j, kb * kBK, full_bar(s));
          }
          ++g;
        }
      }
      // Every load this thread issued has landed before the CTA may exit.
      const uint32_t first = g > (uint32_t)STAGES ? g - STAGES : 0u;
      for (uint32_t i = first; i < g; ++i) mbar_wait_drain(full_bar(i % STAGES), (i / STAGES) & 1u, kDrainNs);
    }
    __syncwarp();  // lanes 1..31 wait here, so the warp reaches the CTA barrier converged
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, BN, !B_KMAJOR);
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
            if (!mbar_wait(full_bar(s), ph, abort_flag, p.err, p.wait_limit_ns)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t a0 = sA + s * kABytes;
            const uint32_t b0 = sB + s * Cfg::kBBytes;
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              // K-major, 128-byte swizzle: rows 128 B apart, 8-row atoms
              // 1024 B apart; one MMA step of K = 16 is 32 bytes along a row.
              const uint64_t ad = smem_desc_sw128(a0 + k * 32, 16, 1024);
              // MN-major B: 64-wide N chunks kBK*128 B apart (LBO), 8-row
              // K groups 1024 B apart (SBO); a K step of 16 rows is 2048 B.
              const uint64_t bd = B_KMAJOR ? smem_desc_sw128(b0 + k * 32, 16, 1024)
                                           : smem_desc_sw128(b0 + k * 2048, kBK * 128, 1024);
              tc_mma_bf16(d_tmem, ad, bd, idesc, (kb > kb_s || k > 0) ? 1u : 0u);
            }
            tc_commit(empty_bar(s));  // stage s is free once these MMAs finish
            ++g;
          }
          if (!ok) break;
          tc_commit(accf_bar(b));  // accumulator b is ready for the epilogue
          ++acc_cnt;
        }
      }
      // All MMAs complete before TMEM is released.
      tc_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0, kDrainNs);
    }
    __syncwarp();
  } else {
    // --------------------------------------------------------- epilogue
    constexpr int CPT = Cfg::kColsPerThread;
    const int ew = warp - 2;
    const int quad = warp & 3;  // a warp may only touch TMEM lanes 32*(warp%4) ..
    const int colpart = ew >> 2;
    const int row_in_tile = quad * 32 + lane;
    const bool ws_vec = (p.N & 3) == 0;
    const uint32_t ebuf = base + Cfg::kEpiOffset + ew * Cfg::kEpiWarpBytes;
    uint32_t acc_cnt = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < num_units; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      const bool split = w.part != 0;                  // partials of this unit, not C
      const bool tail = split && p.tail_splits > 0;    // ... of a split-tail tile
      const int uo = tail ? tail_out : out_tma;
      const CUtensorMap *om = tail ? &tmWs : &tmOut;
      // partial coordinates: a split-tail tile's partials are a compact
      // block (origin px, py of the matrix; rows of pn words), split-K
      // partials whole planes of C's shape
      const int px = tail ? w.tn * BN : 0;
      const int py = tail ? (w.tm - w.slot) * kBM : 0;
      const int pn = tail ? BN : p.N;
      const int64_t pm = tail ? (int64_t)(p.tiles_m * p.tiles_n - p.tail_first) * kBM : (int64_t)p.M;
      const int64_t row = (int64_t)w.tm * kBM + row_in_tile;
      const bool row_ok = row < p.M;
      const int col0 = w.tn * BN + colpart * CPT;
      const int y0 = w.tm * kBM + quad * 32;  // first row of this warp's blocks
      if constexpr (EPI == kEpiS32) {
        if (w.kb1 - w.kb0 <= p.slab_kb) {
          // One slab (K of the unit <= 1024): its exact fp32 sums are the
          // result, streamed 32 columns at a time as in the bf16 epilogue
          // instead of being gathered into int32 registers.
          const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
          if (!__all_sync(0xffffffffu, mbar_wait(accf_bar(b), aph, abort_flag, p.err, p.wait_limit_ns))) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t t0 = tmem_base + b * BN + ((uint32_t)(quad * 32) << 16) + colpart * CPT;
          uint32_t *wrow = split ? reinterpret_cast<uint32_t *>(p.ws) + ((int64_t)w.split * pm + (row - py)) * pn
                                 : nullptr;
#pragma unroll 1
          for (int c = 0; c < CPT / 32; ++c) {
            uint32_t v[32];
            tmem_ld<32>(t0 + c * 32, v);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = static_cast<uint32_t>(__float2int_rn(__uint_as_float(v[i])));
            store_s32_chunk(p, om, ebuf, lane, uo, v, col0 + c * 32, y0, w.split, row_ok, row, wrow, ws_vec, px, py, pn);
          }
          if constexpr (CPT % 32 != 0) {  // a 16-column tail: each lane stores its row
            constexpr int kTail = (CPT / 32) * 32;
            uint32_t v[16];
            tmem_ld<16>(t0 + kTail, v);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = static_cast<uint32_t>(__float2int_rn(__uint_as_float(v[i])));
            if (row_ok) {
              if (split)
                store_words<16>(wrow, col0 + kTail - px, pn, ws_vec, v);
              else
                store_s8_result<16>(p, row, col0 + kTail, v);
            }
          }
          tc_fence_before_sync();
          mbar_arrive(acce_bar(b));
          ++acc_cnt;
          continue;
        }
        int32_t acc[CPT];
#pragma unroll
        for (int i = 0; i < CPT; ++i) acc[i] = 0;
        for (int kb_s = w.kb0; kb_s < w.kb1; kb_s += p.slab_kb) {
          const uint32_t b = acc_cnt & 1u, aph = (acc_cnt >> 1) & 1u;
          // all lanes agree (and reconverge) before the warp-wide TMEM loads
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
          mbar_arrive(acce_bar(b));
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
        mbar_arrive(acce_bar(b));
        ++acc_cnt;
      }
    }
  }

  if (TMA_OUT && warp >= 2 && lane == 0) bulk_wait_all();  // this warp's TMA stores have landed
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

}  // namespace gb300

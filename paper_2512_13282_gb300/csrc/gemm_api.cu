// gemm_api.cu -- the C ABI (include/gb300_gemm.h): argument checks, tile
// and split-K selection, operand staging, TMA descriptor encoding, launches.
//
// One compiled design serves every problem size: as in the paper
// (Sec. 5.3.1), only the tile counts and the number of K steps change from
// one GEMM to the next, and those are runtime kernel arguments here.
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "gb300_gemm.h"
#include "gemm_internal.h"
#include "plan_table.h"

using namespace gb300;

// Device error word (element 0): kernels record kDevErrTimeout here when a
// bounded wait expires; read and cleared by gemm_device_status().  Element 1
// is the sink of the read-bandwidth diagnostic.
__device__ uint32_t g_gemm_dev_err[2] = {0u, 0u};

namespace {

constexpr int kMaxDevices = 64;
constexpr int64_t kMaxExactK = 131071;  // 131072 * 2^14 = 2^31 overflows int32

// Scratch of a call: operand staging copies, split-K partials, and the
// small-M kernel's zeroed ticket counters.  Each stream that calls the
// library on a device gets a scratch slot of its own (the first
// kStreamSlots streams), kept between calls and grown stream-ordered on that
// stream, so that calls on different streams never share device memory; a
// call on a further stream allocates its scratch stream-ordered and frees it
// at its end.
constexpr int kStreamSlots = 16;
struct Scratch {
  bool owned = false;
  cudaStream_t owner = nullptr;
  void *ws = nullptr;
  size_t ws_bytes = 0;
  uint32_t *tickets = nullptr;  // zeroed counters of the small-M kernel
  size_t tickets_count = 0;
  // Once a call has been captured into a CUDA graph, the graph refers to
  // this scratch: buffers replaced by growth are then kept (not freed) until
  // gemm_release_resources(), so that the graph stays valid.
  bool captured = false;
  std::vector<void *> retired;
};

struct DeviceState {
  bool ready = false;
  int sms = 0;
  uint32_t *err = nullptr;
  Scratch slots[kStreamSlots];
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::atomic<uint64_t> g_launches{0};
cudaEvent_t g_prof_start = nullptr, g_prof_stop = nullptr;

}  // namespace

namespace {

// Test and benchmark overrides of the planner, read from the environment
// once (at the first call) and again by gemm_reload_overrides():
// GB300_GEMM_BN (64, 96, 128, 192, 224 or 256; 64 and 96 for bf16 only)
// forces the tile width,
// GB300_GEMM_PAIR (0 or 1) the kernel family, GB300_GEMM_SPLITS (>= 1) the
// split-K factor, GB300_GEMM_TAIL_SPLITS (0, or >= 2) the split tail of
// the tensor-core kernels, GB300_GEMM_SKINNY_MAX_M the largest M sent to the
// CUDA-core kernel, GB300_GEMM_TMA_STORE=0 direct stores (and scalar atomic
// adds for the small-operand kernel's split-K), GB300_GEMM_PDL=0
// plain stream ordering, GB300_GEMM_S8TM=0 the general int8 path for
// small-operand shapes, GB300_GEMM_TINY_MAX_MACS the largest
// int8 problem (M * N * K) sent to the one-launch CUDA-core kernel (0
// disables it), GB300_GEMM_DEBUG=1 prints each plan.
struct Overrides {
  int bn = 0;            // 0: planner's choice
  int pair = -1;         // -1: planner's choice
  int splits = 0;        // 0: planner's choice
  int tail_splits = -1;  // -1: planner's choice, 0: no split tail, >= 2: that split tail where one exists
  int skinny_max_m = -1; // -1: built-in limit
  bool tma_store = true;
  bool pdl = true;
  bool s8tm = true;
  int64_t tiny_max_macs = -1;  // -1: built-in limit
  bool debug = false;
};

int env_int(const char *name, int dflt) {
  const char *s = std::getenv(name);
  return s ? std::atoi(s) : dflt;
}

Overrides read_overrides() {
  Overrides o;
  o.bn = env_int("GB300_GEMM_BN", 0);
  o.pair = env_int("GB300_GEMM_PAIR", -1);
  o.splits = env_int("GB300_GEMM_SPLITS", 0);
  o.tail_splits = env_int("GB300_GEMM_TAIL_SPLITS", -1);
  o.skinny_max_m = env_int("GB300_GEMM_SKINNY_MAX_M", -1);
  o.tma_store = env_int("GB300_GEMM_TMA_STORE", 1) != 0;
  o.pdl = env_int("GB300_GEMM_PDL", 1) != 0;
  o.s8tm = env_int("GB300_GEMM_S8TM", 1) != 0;
  if (const char *t = std::getenv("GB300_GEMM_TINY_MAX_MACS")) o.tiny_max_macs = std::atoll(t);
  o.debug = env_int("GB300_GEMM_DEBUG", 0) != 0;
  return o;
}

std::mutex g_ovr_mu;
Overrides g_ovr;
bool g_ovr_loaded = false;

// The overrides in force (a copy, so that a concurrent reload cannot tear it).
Overrides overrides() {
  std::lock_guard<std::mutex> lk(g_ovr_mu);
  if (!g_ovr_loaded) {
    g_ovr = read_overrides();
    g_ovr_loaded = true;
  }
  return g_ovr;
}

}  // namespace

bool gb300::pdl_enabled() { return overrides().pdl; }

namespace {

uint64_t wait_limit_ns() {
  static uint64_t v = [] {
    const char *s = std::getenv("GB300_GEMM_WAIT_LIMIT_MS");
    const double ms = s ? std::atof(s) : 2000.0;
    return (uint64_t)((ms > 0 ? ms : 2000.0) * 1e6);
  }();
  return v;
}

gemm_status_t device_state(DeviceState **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return GEMM_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceState &d = g_dev[dev];
  if (!d.ready) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return GEMM_ERR_CUDA;
    if (major != 10 || minor != 3) return GEMM_ERR_UNSUPPORTED;  // built for sm_103a only
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&d.err), g_gemm_dev_err) != cudaSuccess)
      return GEMM_ERR_CUDA;
    if (!g_encode) {
      cudaDriverEntryPointQueryResult q;
      void *fn = nullptr;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || !fn)
        return GEMM_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    d.sms = sms;
    d.ready = true;
  }
  *out = &d;
  return GEMM_OK;
}

// The scratch of the call in progress on this host thread (set by ScratchLease).
thread_local Scratch *t_scratch = nullptr;

// Holds the calling stream's scratch for the duration of one call: its own
// slot, or (more streams than slots) a scratch of this call alone, freed
// stream-ordered when the call ends.
class ScratchLease {
 public:
  ScratchLease(DeviceState &d, cudaStream_t st) : st_(st) {
    {
      std::lock_guard<std::mutex> lk(g_mu);
      for (Scratch &x : d.slots)
        if (x.owned && x.owner == st) {
          s_ = &x;
          break;
        }
      if (!s_)
        for (Scratch &x : d.slots)
          if (!x.owned) {
            x.owned = true;
            x.owner = st;
            s_ = &x;
            break;
          }
    }
    if (!s_) s_ = &temp_;
    t_scratch = s_;
  }
  ~ScratchLease() {
    if (s_ == &temp_) {
      if (temp_.ws) cudaFreeAsync(temp_.ws, st_);
      if (temp_.tickets) cudaFreeAsync(temp_.tickets, st_);
    }
    t_scratch = nullptr;
  }
  ScratchLease(const ScratchLease &) = delete;
  ScratchLease &operator=(const ScratchLease &) = delete;

 private:
  cudaStream_t st_;
  Scratch *s_ = nullptr;
  Scratch temp_;
};

// Whether `st` is being captured into a CUDA graph.
bool capturing(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  return cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs != cudaStreamCaptureStatusNone;
}

// Scratch of a stream's own slot needed by a call being captured into a
// CUDA graph: it must exist already (the stream has run a call at least as
// large before the capture), since memory allocated inside the capture
// would belong to the graph alone.  (A stream without a slot of its own --
// more streams than slots -- allocates inside the graph and frees there,
// which the graph owns.)
gemm_status_t scratch_for_capture(Scratch &s, bool enough) {
  if (!enough) return GEMM_ERR_UNSUPPORTED;
  s.captured = true;
  return GEMM_OK;
}

// Release a buffer replaced by growth: stream-ordered, or kept while a
// captured graph may still refer to it.
gemm_status_t retire(Scratch &s, void *p, cudaStream_t st) {
  if (!p) return GEMM_OK;
  if (s.captured) {
    s.retired.push_back(p);
    return GEMM_OK;
  }
  return cudaFreeAsync(p, st) == cudaSuccess ? GEMM_OK : GEMM_ERR_CUDA;
}

// Grow the current call's workspace (stream-ordered, on its own stream) to
// at least `bytes`; the result is scratch_ws().
gemm_status_t ensure_workspace(size_t bytes, cudaStream_t st) {
  Scratch &s = *t_scratch;
  if (capturing(st) && s.owned) return scratch_for_capture(s, bytes <= s.ws_bytes);
  if (bytes <= s.ws_bytes) return GEMM_OK;
  if (s.ws) {
    if (retire(s, s.ws, st) != GEMM_OK) return GEMM_ERR_CUDA;
    s.ws = nullptr;
    s.ws_bytes = 0;
  }
  const size_t grown = bytes + bytes / 4;
  if (cudaMallocAsync(&s.ws, grown, st) != cudaSuccess) {
    s.ws = nullptr;
    return GEMM_ERR_CUDA;
  }
  s.ws_bytes = grown;
  return GEMM_OK;
}
void *scratch_ws() { return t_scratch->ws; }

// Grow the current call's zeroed ticket counters of the small-M kernel to
// `count` (the kernel leaves them zero again).
gemm_status_t ensure_tickets(size_t count, cudaStream_t st) {
  Scratch &s = *t_scratch;
  if (capturing(st) && s.owned) return scratch_for_capture(s, count <= s.tickets_count);
  if (count <= s.tickets_count) return GEMM_OK;
  if (retire(s, s.tickets, st) != GEMM_OK) return GEMM_ERR_CUDA;
  s.tickets = nullptr;
  s.tickets_count = 0;
  const size_t n = count < 1024 ? 1024 : count;
  if (cudaMallocAsync(reinterpret_cast<void **>(&s.tickets), n * sizeof(uint32_t), st) != cudaSuccess ||
      cudaMemsetAsync(s.tickets, 0, n * sizeof(uint32_t), st) != cudaSuccess) {
    s.tickets = nullptr;
    return GEMM_ERR_CUDA;
  }
  s.tickets_count = n;
  return GEMM_OK;
}
uint32_t *scratch_tickets() { return t_scratch->tickets; }

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// GEMM_ERR_CUDA, reporting the failing step (and CUDA's message) on stderr
// when GB300_GEMM_DEBUG=1.
gemm_status_t cuda_failed(const char *what, cudaError_t e = cudaSuccess) {
  if (overrides().debug)
    std::fprintf(stderr, "[gb300_gemm] %s failed%s%s\n", what, e != cudaSuccess ? ": " : "",
                 e != cudaSuccess ? cudaGetErrorString(e) : "");
  return GEMM_ERR_CUDA;
}

// 2-D bf16 tensor map: inner extent `inner` (contiguous), outer extent
// `outer`, row pitch `ld` elements, box box_inner x box_outer, 128-byte
// swizzle.  Out-of-range box elements read as zero.
bool encode_bf16_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t ld,
                    uint32_t box_inner, uint32_t box_outer) {
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {ld * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
                  estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D (C) or 3-D (split-K partials: N x M x splits) tensor map for the
// epilogue's TMA stores: boxes of box_cols columns x 32 rows (x 1 split).
bool encode_out(CUtensorMap *map, CUtensorMapDataType type, uint32_t esize, const void *base, uint64_t N,
                uint64_t M, uint64_t ld, uint64_t splits, uint32_t box_cols = 32) {
  const cuuint64_t dims[3] = {N, M, splits};
  const cuuint64_t strides[2] = {ld * esize, ld * esize * M};
  const cuuint32_t box[3] = {box_cols, 32, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  // 128-, 64- or 32-byte box rows, swizzled to match the staging blocks
  const uint32_t row_bytes = box_cols * esize;
  const CUtensorMapSwizzle sw = row_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : row_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                  : CU_TENSOR_MAP_SWIZZLE_32B;
  return g_encode(map, type, splits > 1 ? 3 : 2, const_cast<void *>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

gemm_status_t check_common(int64_t M, int64_t N, int64_t K, const void *A, int64_t lda, const void *B,
                           int64_t ldb, int layout, const void *C, int64_t ldc) {
  if (M < 0 || N < 0 || K < 0) return GEMM_ERR_INVALID_ARG;
  if (layout != GEMM_B_ROW_MAJOR_KxN && layout != GEMM_B_COL_MAJOR_NxK) return GEMM_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return GEMM_OK;
  if (!C || ldc < N) return GEMM_ERR_INVALID_ARG;
  if (K > 0) {
    if (!A || !B || lda < K) return GEMM_ERR_INVALID_ARG;
    if (layout == GEMM_B_ROW_MAJOR_KxN ? ldb < N : ldb < K) return GEMM_ERR_INVALID_ARG;
  }
  // Index arithmetic inside the kernels uses int for tile and K-block
  // counters and TMA coordinates: keep every extent below 2^31.
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return GEMM_ERR_UNSUPPORTED;
  return GEMM_OK;
}

struct Plan {
  TcVariant v;
  TcParams p;
  int grid;
  double model_us;  // modelled time of the tensor-core kernel (and split-K reduction)
};

// Kernel family, tile width, split-K factor and grid for an M x N x K
// problem on `sms` SMs and `pairs` co-resident SM pairs.
//
// The GB300 counterpart of the paper's balanced-tile search (Sec. 4.5).
// Every candidate -- one CTA per 128 x BN tile or a CTA pair per 256 x BN
// tile, BN among the compiled widths, K split S ways -- runs in
// ceil(tiles * S / slots) rounds of one unit per slot (an SM or an SM pair);
// its modelled time is
//   rounds * (kb_per_unit * kstep + unit) + split terms
// (Eq. 9 with wave quantisation), with the per-variant K-step and unit costs
// and the split constants fitted to measurements on GB300 (plan_table.h,
// generated by tile_model.py).  Plans are ranked by that time plus the share
// kMemWeight of the DRAM time of Eq. 6-8 and 10 (dram_us) that the kernels
// do not hide: with the 129 MB L2 supplying the reuse it separates plans
// only where B is re-read once per group of row tiles (B does not stay in
// L2 beside A and C), which CTA pairs do half as often.  The least rank
// wins; on a tie the earlier candidate (single CTA before pair, wider before
// narrower, fewer splits before more).  tile_model.choose_plan is the same
// rule.
//
// A plan is costed by the work of its busiest CTA -- `steps` K steps in
// `rounds` units -- and, when it writes split-K partials, the reduction
// launch and the partials' bytes: tiles x splits units give rounds =
// ceil(units / slots) of kb_per steps each; a split tail (the tiles of a
// last, partly filled round split in tail_splits) gives the full rounds of
// whole tiles plus one round of a tail unit's steps.
double modelled_us(bool int8, bool pair, int bn, int64_t steps, int64_t rounds, double partial_mb) {
  const int wi = bn == 64 ? 0 : bn == 96 ? 1 : bn == 128 ? 2 : bn == 192 ? 3 : bn == 224 ? 4 : 5;
  const plan_table::StepCost c = plan_table::kCost[int8 ? 1 : 0][pair ? 1 : 0][wi];
  double t = (double)steps * c.kstep_us + (double)rounds * c.unit_us;
  if (partial_mb > 0)
    t += plan_table::kSplitFixedUs[int8 ? 1 : 0] + plan_table::kSplitUsPerMB[int8 ? 1 : 0] * partial_mb;
  return t;
}

// Eq. 6-8 and 10: DRAM bytes of A (once: the grouped raster keeps a group's
// 8 row tiles of A in L2 while it sweeps N), B (once if it fits in half the
// L2 or A, B and C together fit in L2 -- C passes through L2 as the tiles
// store it -- else once per group of 8 row tiles) and C, at the copy
// bandwidth, in microseconds.
double dram_us(int64_t M, int64_t N, int64_t K, bool int8, bool pair) {
  const double a_bytes = 2.0 * M * K, b_bytes = 2.0 * K * N, c_bytes = (double)M * N * (int8 ? 4 : 2);
  double rb = 1.0;
  if (!(b_bytes <= plan_table::kL2Bytes / 2 || a_bytes + b_bytes + c_bytes <= plan_table::kL2Bytes)) {
    rb = (double)ceil_div(M, 8 * (pair ? 2 * kBM : kBM));
    if (rb < 1.0) rb = 1.0;
  }
  return (a_bytes + b_bytes * rb + c_bytes) / (plan_table::kHbmGBs * 1e3);
}

Plan make_plan(int64_t M, int64_t N, int64_t K, bool b_kmajor, int epi, int sms, int pairs,
               bool allow_tail = true) {
  Plan pl{};
  // compiled widths, widest first: the bf16 single-CTA kernels also come 64
  // and 96 wide (96 for B column-major only), for memory-bound GEMMs with
  // few rows
  static const int kWidthsKMajor[] = {256, 224, 192, 128, 96, 64};
  static const int kWidthsMNMajor[] = {256, 192, 128, 64};
  static const int kPairWidthsMNMajor[] = {256, 128};
  const Overrides ovr = overrides();
  const bool int8 = epi == kEpiS32;
  const int64_t num_kb = ceil_div(K, kBK);
  bool best_pair = false;
  int best_bn = 128;
  int64_t best_splits = 1, best_tail = 0, best_kb_tail = 0;
  double best_cost = -1.0, best_model = 0.0;
  const double mem_rank = plan_table::kMemWeight;
  auto consider = [&](bool pair, int bn, int64_t splits, int64_t tail_splits, int64_t kb_tail, double model) {
    const double cost = model + mem_rank * dram_us(M, N, K, int8, pair);
    if (best_cost < 0 || cost < best_cost - 1e-9) {
      best_cost = cost;
      best_model = model;
      best_pair = pair;
      best_bn = bn;
      best_splits = splits;
      best_tail = tail_splits;
      best_kb_tail = kb_tail;
    }
  };
  // A forced tail split (GB300_GEMM_TAIL_SPLITS >= 2) searches the split-tail
  // plans alone first, and all plans only if none exists.
  const bool tail_only_first = allow_tail && ovr.tail_splits >= 2;
  for (int pass = tail_only_first ? 0 : 1; pass < 2 && best_cost < 0; ++pass) {
    const bool tail_only = pass == 0;
    for (int fam = 0; fam < 2; ++fam) {
      const bool pair = fam == 1;
      if (pair && (M <= kBM || pairs <= 0)) continue;  // the second CTA would only compute padding
      if (ovr.pair >= 0 && (ovr.pair != 0) != pair) continue;
      const int *widths = b_kmajor ? kWidthsKMajor : (pair ? kPairWidthsMNMajor : kWidthsMNMajor);
      const bool narrow = !pair && !int8;
      const int nw = b_kmajor ? (narrow ? 6 : 4) : (pair ? 2 : (narrow ? 4 : 3));
      const int64_t slots = pair ? pairs : sms;
      const int64_t tiles_m = ceil_div(M, pair ? 2 * kBM : kBM);
      for (int i = 0; i < nw; ++i) {
        const int bn = widths[i];
        if (N <= 128 && bn > 128) continue;
        if (ovr.bn > 0 && ovr.bn != bn) continue;
        const int64_t tiles = tiles_m * ceil_div(N, bn);
        int64_t seen[17] = {};
        int nseen = 0;
        for (int64_t s = 1; s <= 16 && !tail_only; ++s) {
          int64_t kb_per = ceil_div(num_kb, s < num_kb ? s : num_kb);
          int64_t s2 = ceil_div(num_kb, kb_per);
          if (ovr.splits >= 1) {  // forced: exactly that split
            if (s > 1) break;
            const int64_t f = ovr.splits < num_kb ? ovr.splits : num_kb;
            kb_per = ceil_div(num_kb, f);
            s2 = ceil_div(num_kb, kb_per);
          } else {
            bool dup = false;
            for (int j = 0; j < nseen; ++j) dup = dup || seen[j] == s2;
            if (dup) continue;
            if (s2 > 1 && (kb_per < 4 || tiles * s2 > 2 * slots)) continue;
          }
          seen[nseen++] = s2;
          const int64_t rounds = ceil_div(tiles * s2, slots);
          consider(pair, bn, s2, 0, 0,
                   modelled_us(int8, pair, bn, rounds * kb_per, rounds, s2 > 1 ? 4.0 * s2 * M * N / 1e6 : 0.0));
        }
        // Split tail: whole tiles for the full rounds, the last round's
        // tiles (at most half a round of them) split in S so that they fill
        // it; S = 2 .. 8 with at least 4 K steps a unit.
        const int64_t full = tiles / slots, tail = tiles - full * slots;
        if (!allow_tail || ovr.tail_splits == 0 || ovr.splits > 1 || full < 1 || tail == 0) continue;
        for (int64_t st2 = 2; st2 <= 8 && tail * st2 <= slots; ++st2) {
          if (ovr.tail_splits >= 2 && st2 != ovr.tail_splits) continue;
          const int64_t kb_tail = ceil_div(num_kb, st2);
          if (ceil_div(num_kb, kb_tail) != st2 || kb_tail < 4) continue;
          const double part_mb = 4.0 * st2 * tail * (pair ? 2 * kBM : kBM) * bn / 1e6;
          consider(pair, bn, 1, st2, kb_tail, modelled_us(int8, pair, bn, full * num_kb + kb_tail, full + 1, part_mb));
        }
      }
    }
  }
  const bool pair = best_pair;
  const int bn = best_bn;
  const int64_t slots = pair ? pairs : sms;
  const int64_t tiles_m = ceil_div(M, pair ? 2 * kBM : kBM);
  const int64_t tiles_n = ceil_div(N, bn);
  const int64_t tiles = tiles_m * tiles_n;
  const int64_t kb_per = ceil_div(num_kb, best_splits);
  const int64_t splits = ceil_div(num_kb, kb_per);
  const int64_t full_rounds = best_tail > 0 ? tiles / slots : 0;
  // Output path: the bf16 224-wide kernels keep a pipeline stage and stage
  // their TMA stores through 1 KB blocks; for int8 at 192/224, TMA stores
  // (4 KB blocks, one stage less) win up to 128 K steps per unit, beyond
  // which the extra stage and direct stores win (measured on GB300: 4096^3
  // and 2048 x 11008 x 4096 faster with TMA stores, 2048 x 4096 x 11008 with
  // the extra stage).
  int tma_out;
  if (epi == kEpiBf16)
    tma_out = pair ? tc2_bf16_tma_out(bn) : tc_bf16_tma_out(bn);
  else
    tma_out = ((bn != 224 && bn != 192) || kb_per <= 128) ? 1 : 0;
  pl.v = TcVariant{bn, b_kmajor, epi, pair, tma_out};
  pl.model_us = best_model;
  TcParams &p = pl.p;
  p.M = (int)M;
  p.N = (int)N;
  p.K = (int)K;
  p.tiles_m = (int)tiles_m;
  p.tiles_n = (int)tiles_n;
  p.num_kb = (int)num_kb;
  p.splits = (int)splits;
  p.kb_per_split = (int)kb_per;
  p.slab_kb = epi == kEpiS32 ? 1024 / kBK : (int)num_kb;
  p.group_m = 8;
  p.out_bits = 32;
  p.out_shift = 0;
  p.tail_first = (int)(full_rounds * slots);
  p.tail_splits = (int)best_tail;
  p.tail_kb_per = (int)best_kb_tail;
  p.ws_tma = 0;
  const int64_t units = best_tail > 0 ? full_rounds * slots + (tiles - full_rounds * slots) * best_tail
                                      : tiles * splits;
  const int64_t used = units < slots ? units : slots;
  pl.grid = (int)(pair ? 2 * used : used);
  if (ovr.debug)
    std::fprintf(stderr,
                 "[gb300_gemm] M=%lld N=%lld K=%lld %s B%s: %s BN=%d%s tiles=%lldx%lld splits=%lld "
                 "tail splits=%lld from tile %d grid=%d model %.1f us (SMs %d, co-resident pairs %d)\n",
                 (long long)M, (long long)N, (long long)K, epi == kEpiS32 ? "int8" : "bf16",
                 b_kmajor ? "col" : "row", pair ? "pair" : "single", bn,
                 tma_out == 2 ? " tma-store-1k" : tma_out ? " tma-store" : "", (long long)tiles_m,
                 (long long)tiles_n, (long long)splits, (long long)best_tail, p.tail_first, pl.grid, best_model, sms,
                 pairs);
  return pl;
}

struct WsLayout {
  size_t a_off = 0, b_off = 0, part_off = 0, total = 0;
};

// Planes of 32-bit partials a plan writes (split-K, or a split tail); 0 when
// C is written directly.
int64_t partial_planes(const TcParams &p) { return p.splits > 1 ? p.splits : p.tail_splits; }

// Rows of one plane of a split tail's compact partials (the tail tiles'
// rows one after the other; row pitch BN).
int64_t tail_rows(const Plan &pl) {
  return (int64_t)(pl.p.tiles_m * pl.p.tiles_n - pl.p.tail_first) * (pl.v.pair ? 2 * kBM : kBM);
}

// Bytes of partials: planes of C's shape for split-K, compact blocks of the
// tail tiles for a split tail.
size_t partial_bytes(const Plan &pl) {
  if (pl.p.splits > 1) return (size_t)pl.p.splits * pl.p.M * pl.p.N * 4;
  if (pl.p.tail_splits > 0) return (size_t)pl.p.tail_splits * tail_rows(pl) * pl.v.bn * 4;
  return 0;
}

// Shared path after staging: encode maps, launch the tcgen05 kernel and the
// split-K reduction.
gemm_status_t run_tc(DeviceState &d, Plan &pl, const uint16_t *A, int64_t lda, const uint16_t *B,
                     int64_t ldb, void *C, int64_t ldc, int esize, void *partials, cudaStream_t st) {
  TcParams &p = pl.p;
  CUtensorMap ta, tb;
  if (!encode_bf16_2d(&ta, A, (uint64_t)p.K, (uint64_t)p.M, (uint64_t)lda, kBK, kBM)) return cuda_failed("A tensor map");
  // K-major B boxes cover the CTA's share of the tile width: all of it, or
  // half of it for a CTA pair.
  const uint32_t b_rows = pl.v.pair ? pl.v.bn / 2 : pl.v.bn;
  const bool ok_b = pl.v.b_kmajor
                        ? encode_bf16_2d(&tb, B, (uint64_t)p.K, (uint64_t)p.N, (uint64_t)ldb, kBK, b_rows)
                        : encode_bf16_2d(&tb, B, (uint64_t)p.N, (uint64_t)p.K, (uint64_t)ldb, 64, kBK);
  if (!ok_b) return cuda_failed("B tensor map");
  p.C = C;
  p.ldc = ldc;
  p.c_vec = aligned16(C) && ((ldc * esize) % 16 == 0);
  p.ws = partials;
  // Epilogue stores through TMA where the output allows it: C with a
  // 16-byte aligned base and pitch whose rows also END on a 16-byte
  // boundary (N * esize a multiple of 16) -- a TMA store clipped at column N
  // still writes the rest of the last 16-byte piece of each row, which for
  // ldc > N lies in the caller's padding (measured on GB300: N = 5 bf16
  // with ldc = 8 had columns 5..7 overwritten); split-K partials when their
  // pitch (N words) is a multiple of 16 bytes.  Other cases store directly
  // (GB300_GEMM_TMA_STORE=0 forces that).
  const bool s32 = pl.v.epi == kEpiS32;
  const bool tma_ok = overrides().tma_store &&
                      (p.splits > 1 ? p.N % 4 == 0 && pl.v.tma_out == 1
                                    : p.c_vec != 0 && ((int64_t)p.N * esize) % 16 == 0);
  // An output that will be stored directly wants the variant with the extra
  // pipeline stage where one exists (int8 at 192 / 224).
  if (!tma_ok && s32 && (pl.v.bn == 192 || pl.v.bn == 224)) pl.v.tma_out = 0;
  CUtensorMap tout = tb, tws = tb;
  p.out_tma = kOutDirect;
  p.ws_tma = 0;
  // a split tail's compact partials go through TMA in the variants with
  // 4 KB staging blocks (their rows, BN words, always end on 16 bytes)
  if (p.tail_splits > 0 && pl.v.tma_out == 1 && overrides().tma_store) {
    if (!encode_out(&tws, s32 ? CU_TENSOR_MAP_DATA_TYPE_INT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, partials,
                    (uint64_t)pl.v.bn, (uint64_t)tail_rows(pl), (uint64_t)pl.v.bn, (uint64_t)p.tail_splits))
      return cuda_failed("tail partials tensor map");
    p.ws_tma = 1;
  }
  if (pl.v.tma_out != 0 && tma_ok) {
    if (p.splits > 1) {
      if (p.N % 4 == 0) {
        if (!encode_out(&tout, s32 ? CU_TENSOR_MAP_DATA_TYPE_INT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, partials,
                        (uint64_t)p.N, (uint64_t)p.M, (uint64_t)p.N, (uint64_t)p.splits))
          return cuda_failed("partials tensor map");
        p.out_tma = kOutTmaWs;
      }
    } else if (p.c_vec) {
      const CUtensorMapDataType type = !s32                ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                       : p.out_bits == 32 ? CU_TENSOR_MAP_DATA_TYPE_INT32
                                       : p.out_bits == 16 ? CU_TENSOR_MAP_DATA_TYPE_UINT16
                                                          : CU_TENSOR_MAP_DATA_TYPE_UINT8;
      if (!encode_out(&tout, type, (uint32_t)esize, C, (uint64_t)p.N, (uint64_t)p.M, (uint64_t)ldc, 1,
                      pl.v.tma_out == 2 ? 16 : 32))
        return cuda_failed("C tensor map");
      p.out_tma = kOutTmaC;
    }
  }
  p.err = d.err;
  p.wait_limit_ns = wait_limit_ns();
  const bool prof = g_prof_start && g_prof_stop;
  if (prof && cudaEventRecord(g_prof_start, st) != cudaSuccess) return GEMM_ERR_CUDA;
  cudaError_t e;
  if (pl.v.pair)
    e = pl.v.epi == kEpiS32 ? launch_tc2_s32(pl.v, ta, tb, tout, tws, p, pl.grid, st)
                            : launch_tc2_bf16(pl.v, ta, tb, tout, tws, p, pl.grid, st);
  else
    e = pl.v.epi == kEpiS32 ? launch_tc_s32(pl.v, ta, tb, tout, tws, p, pl.grid, st)
                            : launch_tc_bf16(pl.v, ta, tb, tout, tws, p, pl.grid, st);
  g_launches.fetch_add(1);
  if (e != cudaSuccess) return cuda_failed(pl.v.pair ? "CTA-pair kernel launch" : "tensor-core kernel launch", e);
  if (prof && cudaEventRecord(g_prof_stop, st) != cudaSuccess) return GEMM_ERR_CUDA;
  const int planes = (int)partial_planes(p);
  if (planes > 0) {
    ReduceTiles rt{0, 0, p.tiles_m, p.tiles_n, p.group_m, pl.v.pair ? 2 * kBM : kBM, pl.v.bn};
    if (p.tail_splits > 0) {  // only the split tail's tiles
      rt.first = p.tail_first;
      rt.count = p.tiles_m * p.tiles_n - p.tail_first;
    }
    e = pl.v.epi == kEpiS32
            ? launch_splitk_reduce_s32(static_cast<const int32_t *>(partials), planes, p.M, p.N, C, ldc,
                                       p.out_bits, p.out_shift, rt, st)
            : launch_splitk_reduce_bf16(static_cast<const float *>(partials), planes, p.M, p.N,
                                        static_cast<uint16_t *>(C), ldc, rt, st);
    g_launches.fetch_add(1);
    if (e != cudaSuccess) return GEMM_ERR_CUDA;
  }
  return GEMM_OK;
}

// Largest int8 problem (M * N * K multiply-adds) computed in one launch on
// the CUDA cores (gemm_tiny.cu) instead of staging + tensor cores: below it
// the launches, not the arithmetic, set the time.
constexpr int64_t kTinyMaxMacs = int64_t(1) << 27;  // 512^3

int64_t tiny_max_macs() {
  const Overrides o = overrides();
  // a forced tile width, family or split asks for the tensor-core kernels
  if (o.bn > 0 || o.pair >= 0 || o.splits >= 1 || o.tail_splits >= 2) return 0;
  return o.tiny_max_macs >= 0 ? o.tiny_max_macs : kTinyMaxMacs;
}

// Largest M sent to the CUDA-core small-M kernel: there every B element is
// used at most a few times and streaming B once is the cost.  Measured on
// GB300 against the tensor-core path (N = 4096..11008, K = 4096): int8
// through dp4a, which also skips the staging pass, wins up to M = 8; bf16,
// accumulating with fp32 FMAs, only up to M = 2.
// GB300_GEMM_SKINNY_MAX_M overrides (0 disables the kernel).
int skinny_max_m(bool int8) {
  const int v = overrides().skinny_max_m;
  if (v >= 0) return v > 16 ? 16 : v;
  return int8 ? 8 : 2;
}

gemm_status_t run_skinny(DeviceState &d, int64_t M, int64_t N, int64_t K, const void *A, int64_t lda,
                         const void *B, int64_t ldb, bool b_kmajor, void *C, int64_t ldc, bool int8,
                         cudaStream_t st, int out_bits = 32, int out_shift = 0) {
  const bool row_b = !b_kmajor;
  SkinnyParams p{};
  const int64_t strips = skinny_geometry((int)M, N, K, int8, row_b, d.sms, &p.kb, &p.ks);
  p.A = A;
  p.lda = lda;
  p.B = B;
  p.ldb = ldb;
  p.C = C;
  p.ldc = ldc;
  p.M = (int)M;
  p.N = N;
  p.K = K;
  p.out_bits = out_bits;
  p.out_shift = out_shift;
  const int esize = int8 ? 1 : 2;
  const uint64_t bits = reinterpret_cast<uintptr_t>(B) | (uint64_t)(ldb * esize) | 16u;
  p.b_align = (int)(bits & (~bits + 1));  // lowest set bit: 1, 2, 4, 8 or 16
  gemm_status_t s;
  if (p.ks > 1) {
    if ((s = ensure_workspace((size_t)p.ks * M * N * 4, st)) != GEMM_OK) return s;
    if ((s = ensure_tickets((size_t)strips, st)) != GEMM_OK) return s;
    p.ws = scratch_ws();
    p.tickets = scratch_tickets();
  }
  const bool prof = g_prof_start && g_prof_stop;
  if (prof && cudaEventRecord(g_prof_start, st) != cudaSuccess) return GEMM_ERR_CUDA;
  g_launches.fetch_add(1);
  if (launch_skinny(p, int8, row_b, strips, st) != cudaSuccess) return GEMM_ERR_CUDA;
  if (prof && cudaEventRecord(g_prof_stop, st) != cudaSuccess) return GEMM_ERR_CUDA;
  return GEMM_OK;
}

}  // namespace

extern "C" {

gemm_status_t gemm_bf16_f32acc_bf16(int64_t M, int64_t N, int64_t K, const uint16_t *A, int64_t lda,
                                    const uint16_t *B, int64_t ldb, int b_layout, uint16_t *C,
                                    int64_t ldc, gemm_stream_t stream) {
  gemm_status_t s = check_common(M, N, K, A, lda, B, ldb, b_layout, C, ldc);
  if (s != GEMM_OK || M == 0 || N == 0) return s;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  DeviceState *d = nullptr;
  if ((s = device_state(&d)) != GEMM_OK) return s;
  const ScratchLease lease(*d, st);
  if (K == 0) {
    g_launches.fetch_add(1);
    return launch_zero_fill(C, M, N, ldc, 2, d->sms, st) == cudaSuccess ? GEMM_OK : GEMM_ERR_CUDA;
  }
  const bool b_kmajor = b_layout == GEMM_B_COL_MAJOR_NxK;
  if (M <= skinny_max_m(false))
    return run_skinny(*d, M, N, K, A, lda, B, ldb, b_kmajor, C, ldc, false, st);
  Plan pl = make_plan(M, N, K, b_kmajor, kEpiBf16, d->sms, pair_slots());
  // TMA needs 16-byte aligned bases and row pitches; re-pitch an operand
  // that is not, into the workspace.
  const bool pack_a = !(aligned16(A) && (lda * 2) % 16 == 0);
  const bool pack_b = !(aligned16(B) && (ldb * 2) % 16 == 0);
  const int64_t b_rows = b_kmajor ? N : K, b_cols = b_kmajor ? K : N;
  const int64_t lda_p = (K + 7) / 8 * 8, ldb_p = (b_cols + 7) / 8 * 8;
  WsLayout L;
  size_t off = 0;
  if (pack_a) { L.a_off = off; off = align_up(off + (size_t)M * lda_p * 2, 256); }
  if (pack_b) { L.b_off = off; off = align_up(off + (size_t)b_rows * ldb_p * 2, 256); }
  if (partial_planes(pl.p) > 0) {
    L.part_off = off;
    off = align_up(off + partial_bytes(pl), 256);
  }
  L.total = off;
  if (L.total && (s = ensure_workspace(L.total, st)) != GEMM_OK) return s;
  uint8_t *ws = static_cast<uint8_t *>(scratch_ws());
  const uint16_t *Au = A, *Bu = B;
  int64_t lda_u = lda, ldb_u = ldb;
  if (pack_a) {
    uint16_t *dst = reinterpret_cast<uint16_t *>(ws + L.a_off);
    g_launches.fetch_add(1);
    if (launch_pack_u16(A, M, K, lda, dst, lda_p, d->sms, st) != cudaSuccess) return GEMM_ERR_CUDA;
    Au = dst;
    lda_u = lda_p;
  }
  if (pack_b) {
    uint16_t *dst = reinterpret_cast<uint16_t *>(ws + L.b_off);
    g_launches.fetch_add(1);
    if (launch_pack_u16(B, b_rows, b_cols, ldb, dst, ldb_p, d->sms, st) != cudaSuccess) return GEMM_ERR_CUDA;
    Bu = dst;
    ldb_u = ldb_p;
  }
  return run_tc(*d, pl, Au, lda_u, Bu, ldb_u, C, ldc, 2, partial_planes(pl.p) > 0 ? ws + L.part_off : nullptr,
                st);
}

}  // extern "C"

namespace {

// int8 operand streamed by gemm_s8tm_kernel: boxes of 128 bytes x 128 rows
// with the 128-byte swizzle its converter warps expect.  inner = K and
// rows = P's rows for a K-contiguous P; inner = P's rows and rows = K for a
// P stored K x P_rows (read transposed).
bool encode_s8_rows(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows, uint64_t ld) {
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {ld};
  const cuuint32_t box[2] = {128, (cuuint32_t)kBM};
  const cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// K splits of the small-operand int8 kernel.  A unit (one P tile, one
// split) is a chain of k-blocks that each pass the converter, the TMEM store
// and the MMA in turn, ~0.57 us a k-block on GB300 until every SM streams
// (then the P stream's rate takes over), and the CTAs (one per SM) run
// their units one after the other; so the split
// minimises rounds * (k-blocks per unit + kS8tmUnitKb), the per-unit start
// and drain counted in k-blocks, plus kS8tmReduceKb when int16 / int8
// outputs need the reduction launch.  Measured on GB300 (whole GEMM after a
// 512 MiB flush), this picks the fastest of 1-8 splits for int32 outputs on
// 128 x 11008 x 4096 (3 splits: 258 units in two rounds of 11 k-blocks,
// 34.3 -> 30.2 us against one split on 86 SMs), 128 x 12288 x 4096,
// 128 x 4096 x 11008, 128 x 4096 x 4096, 16 x 4096 x 4096 and
// 8192 x 64 x 8192, and for int16 outputs on 128 x 11008 / 12288 x 4096
// (one split: the reduction launch costs more than the shorter chains gain)
// and 128 x 4096 x 4096 (4 splits).  At least 4 k-blocks (of 128) per split,
// at most 16 splits (or the forced count); rounded so that no split is
// empty.
constexpr int64_t kS8tmUnitKb = 2;
constexpr int64_t kS8tmReduceKb = 10;

int64_t s8tm_splits(int64_t tiles, int64_t num_kb, int sms, int forced, bool reduce_launch) {
  if (forced >= 1) {
    const int64_t f = forced < num_kb ? forced : num_kb;
    return ceil_div(num_kb, ceil_div(num_kb, f));
  }
  int64_t best = 1, best_cost = -1;
  for (int64_t s = 1; s <= 16 && s <= num_kb; ++s) {
    const int64_t kb_per = ceil_div(num_kb, s);
    const int64_t s2 = ceil_div(num_kb, kb_per);
    if (s2 != s || (s2 > 1 && kb_per < 4)) continue;  // a count already seen, or too short a split
    const int64_t rounds = ceil_div(tiles * s2, (int64_t)sms);
    const int64_t cost = rounds * (kb_per + kS8tmUnitKb) + (s2 > 1 && reduce_launch ? kS8tmReduceKb : 0);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = s2;
    }
  }
  return best;
}

// Which operand the small-operand int8 kernel streams, if any: P = B with
// M <= 128 (swap), P = A with N <= 128 < M; p_kmajor is false for B stored
// K x N, read transposed.
bool s8tm_shape(int64_t M, int64_t N, bool b_kmajor, bool *swap, bool *p_kmajor) {
  if (M <= kBM && N > kBM)
    *swap = true;
  else if (N <= kBM && M > kBM)
    *swap = false;
  else
    return false;
  *p_kmajor = !*swap || b_kmajor;
  return true;
}

// Memory-bound int8 shapes, where one operand is far larger than the other:
// M <= 128 (the weights, P = B, are streamed as int8 and the activations
// Q = A staged; B stored N x K is read K-major, B stored K x N transposed),
// or N <= 128 with M > 128 (P = A, Q = B, in either layout).
// gemm_s8tm_kernel converts P inside the kernel, so P moves once as int8
// instead of three times as staged bf16.  Returns false, having launched
// nothing, when the shape or P's alignment (16-byte base and pitch, for
// TMA) rules the path out; GB300_GEMM_S8TM=0 turns it off and
// GB300_GEMM_SPLITS forces the split-K factor.
bool try_s8tm(DeviceState &d, int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda, const int8_t *B,
              int64_t ldb, bool b_kmajor, void *C, int64_t ldc, int out_bits, int shift, cudaStream_t st,
              gemm_status_t *status) {
  const Overrides ovr = overrides();
  if (!ovr.s8tm) return false;
  bool swap, p_kmajor;  // p_kmajor false: B stored K x N, P's rows are its k-rows
  if (!s8tm_shape(M, N, b_kmajor, &swap, &p_kmajor)) return false;
  const int8_t *P = swap ? B : A;
  const int64_t ldp = swap ? ldb : lda;
  if (!aligned16(P) || ldp % 16 != 0) return false;
  const int64_t P_rows = swap ? N : M, Q_rows = swap ? M : N;
  const int qn = Q_rows <= 64 ? 64 : 128;
  // Q(q, k): A[q][k] when swapped; else B, stored N x K or K x N.
  const int8_t *Qs = swap ? A : B;
  const int64_t sq = (swap || b_kmajor) ? (swap ? lda : ldb) : 1;
  const int64_t sk = (swap || b_kmajor) ? 1 : ldb;
  const int64_t num_kb = ceil_div(K, kS8tmKB);
  const int64_t tiles_p = ceil_div(P_rows, kBM), tiles_q = ceil_div(Q_rows, qn);
  const int64_t tiles = tiles_p * tiles_q;
  int64_t splits = s8tm_splits(tiles, num_kb, d.sms, ovr.splits, out_bits != 32);
  const int64_t kb_per = ceil_div(num_kb, splits);
  gemm_status_t s;
  // split-K: int32 outputs are added into C (zeroed by the staging launch),
  // int16 / int8 ones go through int32 partials and the reduction kernel
  const bool add_into_c = splits > 1 && out_bits == 32;
  const size_t q_bytes = align_up(s8tm_q_image_bytes(qn, Q_rows, K), 256);
  const size_t total = q_bytes + (splits > 1 && !add_into_c ? (size_t)splits * M * N * 4 : 0);
  if ((s = ensure_workspace(total, st)) != GEMM_OK) {
    *status = s;
    return true;
  }
  uint8_t *ws = static_cast<uint8_t *>(scratch_ws());
  *status = GEMM_ERR_CUDA;
  g_launches.fetch_add(1);
  if (launch_s8tm_stage_q(Qs, sq, sk, Q_rows, K, qn, ws, add_into_c ? static_cast<int32_t *>(C) : nullptr, M, N,
                          ldc, st) != cudaSuccess)
    return true;
  CUtensorMap tp;
  if (!(p_kmajor ? encode_s8_rows(&tp, P, (uint64_t)K, (uint64_t)P_rows, (uint64_t)ldp)
                 : encode_s8_rows(&tp, P, (uint64_t)P_rows, (uint64_t)K, (uint64_t)ldp)))
    return true;
  S8tmParams p{};
  p.P_rows = (int)P_rows;
  p.Q_rows = (int)Q_rows;
  p.K = (int)K;
  p.M = (int)M;
  p.N = (int)N;
  p.tiles_p = (int)tiles_p;
  p.tiles_q = (int)tiles_q;
  p.num_kb = (int)num_kb;
  p.splits = (int)splits;
  p.kb_per_split = (int)kb_per;
  p.slab_kb = 1024 / kS8tmKB;
  p.add_into_c = add_into_c ? 1 : 0;
  p.swap = swap ? 1 : 0;
  p.C = C;
  p.ldc = ldc;
  p.ws = splits > 1 && !add_into_c ? ws + q_bytes : nullptr;
  p.err = d.err;
  p.wait_limit_ns = wait_limit_ns();
  p.out_bits = out_bits;
  p.out_shift = shift;
  p.q_img = ws;
  // Split-K into int32 C by TMA reductions where C's base, pitch and row
  // ends allow TMA (rows ending on a 16-byte boundary: a clipped TMA
  // reduction would touch the rest of the row's last 16-byte piece), else
  // by element-wise atomic adds.
  CUtensorMap tc = tp;
  p.c_tma = 0;
  if (add_into_c && overrides().tma_store && aligned16(C) && (ldc * 4) % 16 == 0 && (N * 4) % 16 == 0) {
    if (!encode_out(&tc, CU_TENSOR_MAP_DATA_TYPE_INT32, 4, C, (uint64_t)N, (uint64_t)M, (uint64_t)ldc, 1))
      return true;
    p.c_tma = 1;
  }
  const int64_t units = tiles * splits;
  const int grid = (int)(units < d.sms ? units : d.sms);
  if (ovr.debug)
    std::fprintf(stderr,
                 "[gb300_gemm] M=%lld N=%lld K=%lld int8 s8tm %s%s QN=%d tiles=%lldx%lld splits=%lld grid=%d\n",
                 (long long)M, (long long)N, (long long)K, swap ? "swap" : "direct", p_kmajor ? "" : " P-transposed",
                 qn, (long long)tiles_p, (long long)tiles_q, (long long)splits, grid);
  const bool prof = g_prof_start && g_prof_stop;
  if (prof && cudaEventRecord(g_prof_start, st) != cudaSuccess) return true;
  g_launches.fetch_add(1);
  if (launch_s8tm(qn, p_kmajor, tp, tc, p, grid, st) != cudaSuccess) return true;
  if (prof && cudaEventRecord(g_prof_stop, st) != cudaSuccess) return true;
  if (splits > 1 && !add_into_c) {
    g_launches.fetch_add(1);
    if (launch_splitk_reduce_s32(static_cast<const int32_t *>(p.ws), (int)splits, M, N, C, ldc, out_bits, shift,
                                 ReduceTiles{}, st) != cudaSuccess)
      return true;
  }
  *status = GEMM_OK;
  return true;
}

// The int8 GEMM behind gemm_s8s8_s32 (out_bits 32), gemm_s8s8_s16 and
// gemm_s8s8_s8 (out_bits 16 / 8, right shift `shift`): the exact int32 sum
// is formed the same way for all three; only the final store differs.
gemm_status_t s8_gemm(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda, const int8_t *B,
                      int64_t ldb, int b_layout, void *C, int64_t ldc, int out_bits, int shift,
                      gemm_stream_t stream) {
  gemm_status_t s = check_common(M, N, K, A, lda, B, ldb, b_layout, C, ldc);
  if (s != GEMM_OK) return s;
  if (shift < 0 || shift > 31) return GEMM_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return GEMM_OK;
  if (K > kMaxExactK) return GEMM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  DeviceState *d = nullptr;
  if ((s = device_state(&d)) != GEMM_OK) return s;
  const ScratchLease lease(*d, st);
  const int out_esize = out_bits / 8;
  if (K == 0) {  // every sum is 0, and 0 requantises to 0
    g_launches.fetch_add(1);
    return launch_zero_fill(C, M, N, ldc, out_esize, d->sms, st) == cudaSuccess ? GEMM_OK : GEMM_ERR_CUDA;
  }
  const bool b_kmajor = b_layout == GEMM_B_COL_MAJOR_NxK;
  if (M <= skinny_max_m(true))
    return run_skinny(*d, M, N, K, A, lda, B, ldb, b_kmajor, C, ldc, true, st, out_bits, shift);
  if ((double)M * (double)N * (double)K <= (double)tiny_max_macs()) {
    const TinyParams tp{A, lda, B, ldb, C, ldc, M, N, K, out_bits, shift};
    const bool prof = g_prof_start && g_prof_stop;
    if (prof && cudaEventRecord(g_prof_start, st) != cudaSuccess) return GEMM_ERR_CUDA;
    g_launches.fetch_add(1);
    if (launch_tiny_s8(tp, !b_kmajor, st) != cudaSuccess) return GEMM_ERR_CUDA;
    if (prof && cudaEventRecord(g_prof_stop, st) != cudaSuccess) return GEMM_ERR_CUDA;
    return GEMM_OK;
  }
  if (try_s8tm(*d, M, N, K, A, lda, B, ldb, b_kmajor, C, ldc, out_bits, shift, st, &s)) return s;
  Plan pl = make_plan(M, N, K, b_kmajor, kEpiS32, d->sms, pair_slots());
  pl.p.out_bits = out_bits;
  pl.p.out_shift = shift;
  // Stage both operands as bf16 (exact for int8) with 16-byte aligned rows.
  const int64_t b_rows = b_kmajor ? N : K, b_cols = b_kmajor ? K : N;
  const int64_t lda_p = (K + 7) / 8 * 8, ldb_p = (b_cols + 7) / 8 * 8;
  WsLayout L;
  size_t off = 0;
  L.a_off = off;
  off = align_up(off + (size_t)M * lda_p * 2, 256);
  L.b_off = off;
  off = align_up(off + (size_t)b_rows * ldb_p * 2, 256);
  if (partial_planes(pl.p) > 0) {
    L.part_off = off;
    off = align_up(off + partial_bytes(pl), 256);
  }
  L.total = off;
  if ((s = ensure_workspace(L.total, st)) != GEMM_OK) return s;
  uint8_t *ws = static_cast<uint8_t *>(scratch_ws());
  uint16_t *Ab = reinterpret_cast<uint16_t *>(ws + L.a_off);
  uint16_t *Bb = reinterpret_cast<uint16_t *>(ws + L.b_off);
  g_launches.fetch_add(1);
  if (launch_s8_to_bf16_pair(S8Job{A, M, K, lda, Ab, lda_p}, S8Job{B, b_rows, b_cols, ldb, Bb, ldb_p}, d->sms,
                             st) != cudaSuccess)
    return GEMM_ERR_CUDA;
  return run_tc(*d, pl, Ab, lda_p, Bb, ldb_p, C, ldc, out_esize,
                partial_planes(pl.p) > 0 ? ws + L.part_off : nullptr, st);
}

}  // namespace

extern "C" {

gemm_status_t gemm_s8s8_s32(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                            const int8_t *B, int64_t ldb, int b_layout, int32_t *C, int64_t ldc,
                            gemm_stream_t stream) {
  return s8_gemm(M, N, K, A, lda, B, ldb, b_layout, C, ldc, 32, 0, stream);
}

gemm_status_t gemm_s8s8_s16(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                            const int8_t *B, int64_t ldb, int b_layout, int16_t *C, int64_t ldc, int shift,
                            gemm_stream_t stream) {
  return s8_gemm(M, N, K, A, lda, B, ldb, b_layout, C, ldc, 16, shift, stream);
}

gemm_status_t gemm_s8s8_s8(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                           const int8_t *B, int64_t ldb, int b_layout, int8_t *C, int64_t ldc, int shift,
                           gemm_stream_t stream) {
  return s8_gemm(M, N, K, A, lda, B, ldb, b_layout, C, ldc, 8, shift, stream);
}

const char *gemm_status_string(gemm_status_t status) {
  switch (status) {
    case GEMM_OK: return "GEMM_OK";
    case GEMM_ERR_INVALID_ARG: return "GEMM_ERR_INVALID_ARG: invalid argument";
    case GEMM_ERR_UNSUPPORTED: return "GEMM_ERR_UNSUPPORTED: unsupported size or device";
    case GEMM_ERR_CUDA: return "GEMM_ERR_CUDA: CUDA call or launch failed";
    case GEMM_ERR_TIMEOUT: return "GEMM_ERR_TIMEOUT: a bounded device wait expired";
  }
  return "unknown gemm_status_t";
}

gemm_status_t gemm_device_status(void) {
  DeviceState *d = nullptr;
  gemm_status_t s = device_state(&d);
  if (s != GEMM_OK) return s;
  if (cudaDeviceSynchronize() != cudaSuccess) return GEMM_ERR_CUDA;
  uint32_t v = 0;
  if (cudaMemcpy(&v, d->err, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return GEMM_ERR_CUDA;
  if (v != 0) {
    const uint32_t zero = 0;
    if (cudaMemcpy(d->err, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return GEMM_ERR_CUDA;
  }
  return v == 0 ? GEMM_OK : static_cast<gemm_status_t>(v);
}

void gemm_release_resources(void) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceState &d = g_dev[dev];
  for (Scratch &x : d.slots) {
    if (x.ws) cudaFree(x.ws);
    if (x.tickets) cudaFree(x.tickets);
    for (void *p : x.retired) cudaFree(p);
    x = Scratch{};
  }
  d.ready = false;  // look the device's symbols up again at the next call
  noalloc_forget_device(dev);
}

uint64_t gemm_launch_count(void) { return g_launches.load(); }

void gemm_reload_overrides(void) {
  const Overrides o = read_overrides();
  std::lock_guard<std::mutex> lk(g_ovr_mu);
  g_ovr = o;
  g_ovr_loaded = true;
}

gemm_status_t gemm_selftest_wait_timeout(uint64_t limit_ns, gemm_stream_t stream) {
  if (limit_ns == 0 || limit_ns > 1000000000ull) return GEMM_ERR_INVALID_ARG;
  DeviceState *d = nullptr;
  gemm_status_t s = device_state(&d);
  if (s != GEMM_OK) return s;
  g_launches.fetch_add(1);
  return launch_wait_timeout_probe(d->err, limit_ns, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? GEMM_OK
             : GEMM_ERR_CUDA;
}

gemm_status_t gemm_plan_query(int64_t M, int64_t N, int64_t K, int int8, int b_layout, int sms, int pair_slots_,
                              gemm_plan_t *out) {
  if (!out || M < 0 || N < 0 || K < 0 || sms <= 0 || pair_slots_ < 0) return GEMM_ERR_INVALID_ARG;
  if (b_layout != GEMM_B_ROW_MAJOR_KxN && b_layout != GEMM_B_COL_MAJOR_NxK) return GEMM_ERR_INVALID_ARG;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX || (int8 && K > kMaxExactK)) return GEMM_ERR_UNSUPPORTED;
  *out = gemm_plan_t{};
  const bool b_kmajor = b_layout == GEMM_B_COL_MAJOR_NxK;
  if (M == 0 || N == 0) {
    out->route = GEMM_ROUTE_NONE;
    return GEMM_OK;
  }
  if (K == 0) {
    out->route = GEMM_ROUTE_ZERO_FILL;
    return GEMM_OK;
  }
  if (M <= skinny_max_m(int8 != 0)) {
    out->route = GEMM_ROUTE_SMALL_M;
    return GEMM_OK;
  }
  if (int8 && (double)M * (double)N * (double)K <= (double)tiny_max_macs()) {
    out->route = GEMM_ROUTE_TINY;
    out->bn = 32;
    out->splits = 1;
    out->grid = (int)(ceil_div(M, 32) * ceil_div(N, 32));
    return GEMM_OK;
  }
  bool swap, p_kmajor;
  // tight leading dimensions: P's pitch is K (K-major) or N (B stored K x N)
  if (int8 && overrides().s8tm && s8tm_shape(M, N, b_kmajor, &swap, &p_kmajor) &&
      (p_kmajor ? K : N) % 16 == 0) {
    const int64_t Q_rows = swap ? M : N, P_rows = swap ? N : M;
    const int qn = Q_rows <= 64 ? 64 : 128;
    const int64_t tiles = ceil_div(P_rows, kBM) * ceil_div(Q_rows, qn);
    const int64_t splits = s8tm_splits(tiles, ceil_div(K, kS8tmKB), sms, overrides().splits, false);
    out->route = GEMM_ROUTE_SMALL_OPERAND;
    out->bn = qn;
    out->splits = (int)splits;
    out->grid = (int)(tiles * splits < sms ? tiles * splits : sms);
    return GEMM_OK;
  }
  const int epi = int8 ? kEpiS32 : kEpiBf16;
  const Plan pl = make_plan(M, N, K, b_kmajor, epi, sms, pair_slots_);
  const int ew = int8 && pl.v.bn != 128 ? 8 : 4;
  out->route = pl.v.pair ? GEMM_ROUTE_TC_PAIR : GEMM_ROUTE_TC_SINGLE;
  out->bn = pl.v.bn;
  out->splits = pl.p.splits;
  out->tail_splits = pl.p.tail_splits;
  out->stages = tc_max_stages(pl.v.pair ? pl.v.bn / 2 : pl.v.bn, ew, pl.v.tma_out);
  out->grid = pl.grid;
  out->model_us = pl.model_us;
  out->dram_us = dram_us(M, N, K, int8 != 0, pl.v.pair);
  return GEMM_OK;
}

gemm_status_t gemm_selftest_read_stream(const void *ptr, size_t bytes, gemm_stream_t stream) {
  if (!ptr || bytes % 16 != 0 || (reinterpret_cast<uintptr_t>(ptr) & 15) != 0) return GEMM_ERR_INVALID_ARG;
  DeviceState *d = nullptr;
  gemm_status_t s = device_state(&d);
  if (s != GEMM_OK) return s;
  g_launches.fetch_add(1);
  // the sink sits beside the error word and is written only for one
  // particular fold of the data
  return launch_read_stream(ptr, bytes, d->err + 1, d->sms, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? GEMM_OK
             : GEMM_ERR_CUDA;
}

void gemm_profile_events(void *start_event, void *stop_event) {
  g_prof_start = static_cast<cudaEvent_t>(start_event);
  g_prof_stop = static_cast<cudaEvent_t>(stop_event);
}

}  // extern "C"

namespace gb300 {

gemm_status_t validate_s8(int64_t M, int64_t N, int64_t K, const void *A, int64_t lda, const void *B,
                          int64_t ldb, int b_layout, const void *C, int64_t ldc) {
  gemm_status_t s = check_common(M, N, K, A, lda, B, ldb, b_layout, C, ldc);
  if (s != GEMM_OK) return s;
  if (M > 0 && N > 0 && K > kMaxExactK) return GEMM_ERR_UNSUPPORTED;
  return GEMM_OK;
}

// The int8 GEMM of gemm_s8s8_s32 with operand staging and split-K partials
// placed in caller-provided device scratch [scratch, scratch + capacity)
// instead of the library's workspace.  Returns GEMM_ERR_UNSUPPORTED, before
// launching anything, when the problem needs more than `capacity` bytes.
gemm_status_t s8_gemm_into_scratch(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                                   const int8_t *B, int64_t ldb, int b_layout, int32_t *C, int64_t ldc,
                                   cudaStream_t st, void *scratch, size_t capacity) {
  gemm_status_t s = validate_s8(M, N, K, A, lda, B, ldb, b_layout, C, ldc);
  if (s != GEMM_OK || M == 0 || N == 0) return s;
  DeviceState *d = nullptr;
  if ((s = device_state(&d)) != GEMM_OK) return s;
  if (K == 0) {
    g_launches.fetch_add(1);
    return launch_zero_fill(C, M, N, ldc, 4, d->sms, st) == cudaSuccess ? GEMM_OK : GEMM_ERR_CUDA;
  }
  const bool b_kmajor = b_layout == GEMM_B_COL_MAJOR_NxK;
  Plan pl = make_plan(M, N, K, b_kmajor, kEpiS32, d->sms, pair_slots());
  const int64_t b_rows = b_kmajor ? N : K, b_cols = b_kmajor ? K : N;
  const int64_t lda_p = (K + 7) / 8 * 8, ldb_p = (b_cols + 7) / 8 * 8;
  const size_t a_off = 0;
  const size_t b_off = align_up((size_t)M * lda_p * 2, 256);
  const size_t part_off = align_up(b_off + (size_t)b_rows * ldb_p * 2, 256);
  auto total_of = [&](const Plan &q) {
    return partial_planes(q.p) > 0 ? align_up(part_off + partial_bytes(q), 256) : part_off;
  };
  // a split tail's partial planes may not fit the caller's scratch: plan
  // without one then
  if (pl.p.tail_splits > 0 && total_of(pl) > capacity)
    pl = make_plan(M, N, K, b_kmajor, kEpiS32, d->sms, pair_slots(), false);
  const size_t total = total_of(pl);
  if (!scratch || total > capacity) return GEMM_ERR_UNSUPPORTED;
  uint8_t *ws = static_cast<uint8_t *>(scratch);
  uint16_t *Ab = reinterpret_cast<uint16_t *>(ws + a_off);
  uint16_t *Bb = reinterpret_cast<uint16_t *>(ws + b_off);
  g_launches.fetch_add(1);
  if (launch_s8_to_bf16_pair(S8Job{A, M, K, lda, Ab, lda_p}, S8Job{B, b_rows, b_cols, ldb, Bb, ldb_p}, d->sms,
                             st) != cudaSuccess)
    return GEMM_ERR_CUDA;
  return run_tc(*d, pl, Ab, lda_p, Bb, ldb_p, C, ldc, 4, partial_planes(pl.p) > 0 ? ws + part_off : nullptr, st);
}

}  // namespace gb300


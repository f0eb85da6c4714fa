/*
 * gb300_gemm.h -- C ABI of the GB300 (sm_103a) dense GEMM library.
 *
 * The operation (Sec. 4.1 of "Striking the Balance: GEMM Performance
 * Optimization Across Generations of Ryzen AI NPUs", arXiv 2512.13282):
 *
 *     C = A . B,   A is M x K, B is K x N, C is M x N,
 *
 * with A and C row-major and B either row-major (K x N) or column-major
 * (stored N x K, K contiguous) (Sec. 4.2.2).  Two precisions (Sec. 5.1,
 * Table 1): "int8-int32" -- int8 operands, exact int32 result -- and
 * "bf16-bf16" -- bf16 operands, float32 accumulation, bf16 result rounded to
 * nearest, ties to even.  Arbitrary M, N, K are supported (Sec. 5.3.1 pads to
 * the design's native size; here partial edge tiles are clipped instead, so
 * nothing outside [0,M) x [0,N) of C is ever written).
 *
 * Conventions shared by every entry point:
 *   - Pointers A, B, C are DEVICE pointers owned by the caller; the library
 *     never frees them.  A, B and C must not overlap.
 *   - Leading dimensions are in elements: row i of A starts at A + i*lda;
 *     row k of a row-major B at B + k*ldb, row j of a column-major B (its
 *     column j) at B + j*ldb; row i of C at C + i*ldc.
 *   - The call is asynchronous on `stream` (0 = legacy default stream): it
 *     validates, enqueues its kernels and returns without synchronising.
 *   - M == 0 or N == 0 is a no-op returning GEMM_OK; K == 0 writes zeros.
 *   - Errors are returned as status codes; nothing is thrown across the ABI.
 *   - The library keeps lazily grown device scratch (operand staging copies,
 *     split-K partials, the small-M kernel's counters), allocated
 *     stream-ordered on first need, one set per stream: the first 16 streams
 *     that call the library on a device keep theirs between calls, a call on
 *     any further stream allocates its own and frees it (stream-ordered) when
 *     it ends.  Calls on different streams may therefore run concurrently;
 *     calls on one stream must not be issued from several host threads at
 *     once.  gemm_release_resources() frees the scratch.
 *   - CUDA graphs: calls may be captured on a stream that has already run,
 *     outside capture, calls needing at least as much scratch (the same
 *     shapes, say); a captured call that would need more returns
 *     GEMM_ERR_UNSUPPORTED before enqueuing anything.  Scratch that a graph
 *     refers to stays allocated until gemm_release_resources(), after which
 *     graphs captured before must not be launched.
 *   - Environment variables that override the planner, for tests and
 *     benchmarks (int8 results are identical either way; bf16 results may
 *     differ in summation order, within the same accuracy): GB300_GEMM_BN,
 *     GB300_GEMM_PAIR, GB300_GEMM_SPLITS, GB300_GEMM_TAIL_SPLITS (0: no
 *     split tail; S >= 2: split the last round's tiles in S where the plan
 *     has such a round), GB300_GEMM_SKINNY_MAX_M,
 *     GB300_GEMM_TMA_STORE=0 (results stored, and split-K sums added into
 *     C, element by element instead of by TMA), GB300_GEMM_PDL=0 (plain
 *     stream ordering between the library's kernels), GB300_GEMM_S8TM=0 (int8
 *     GEMMs with one operand of at most 128 rows take the general path
 *     instead of converting the large operand inside the kernel),
 *     GB300_GEMM_TINY_MAX_MACS (largest M*N*K of an int8 GEMM computed in one
 *     launch on the CUDA cores; 0 disables that kernel, and so does forcing
 *     a tile width, family or split with the variables above) and
 *     GB300_GEMM_DEBUG=1 (prints each plan to stderr).  They are read once,
 *     at the first call, and again by gemm_reload_overrides().
 *     GB300_GEMM_WAIT_LIMIT_MS (read once) bounds every device-side wait
 *     (default 2000 ms).
 */
#ifndef GB300_GEMM_H
#define GB300_GEMM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif
/* The library is built with hidden symbols by default; these are its exports. */
#if defined(__GNUC__)
#pragma GCC visibility push(default)
#endif

typedef struct CUstream_st *gemm_stream_t; /* same object as cudaStream_t */

typedef enum {
  GEMM_OK = 0,
  GEMM_ERR_INVALID_ARG = 1, /* negative size, null pointer with nonzero extent,
                               lda < K, ldb < N (row-major) or < K (column-major),
                               ldc < N, unknown layout flag */
  GEMM_ERR_UNSUPPORTED = 2, /* int8 with K > 131071: 131072 * (-128)^2 = 2^31 no
                               longer fits int32, so exactness is not possible;
                               or a device that is not sm_103 */
  GEMM_ERR_CUDA = 3,        /* a CUDA runtime/driver call or launch failed */
  GEMM_ERR_TIMEOUT = 4      /* a bounded on-device wait expired; reported by
                               gemm_device_status() after the stream is synced */
} gemm_status_t;

typedef enum {
  GEMM_B_ROW_MAJOR_KxN = 0, /* B(k, n) = B[k*ldb + n] */
  GEMM_B_COL_MAJOR_NxK = 1  /* B(k, n) = B[n*ldb + k] */
} gemm_b_layout_t;

/*
 * int8-int32 (Sec. 5.1, Table 1): C[i][j] = sum_k A[i][k] * B(k, j), exact.
 *   A: int8, M x K row-major (lda >= K).  B: int8, layout per b_layout.
 *   C: int32, M x N row-major (ldc >= N), fully overwritten in [0,M) x [0,N).
 *   K <= 131071 guarantees the exact sum fits int32; larger K returns
 *   GEMM_ERR_UNSUPPORTED.
 */
gemm_status_t gemm_s8s8_s32(int64_t M, int64_t N, int64_t K,
                            const int8_t *A, int64_t lda,
                            const int8_t *B, int64_t ldb, int b_layout,
                            int32_t *C, int64_t ldc, gemm_stream_t stream);

/*
 * int8-int16 and int8-int8 (Sec. 5.1, Tables 1-3: int8 GEMMs whose output
 * precision is reduced to 16 or 8 bits).  The paper gives no rounding rule;
 * this library's is:
 *   C[i][j] = saturate_T(round_half_even(S_ij / 2^shift)),
 * S_ij = sum_k a_ik * b_kj the exact sum of gemm_s8s8_s32, T = int16 or int8
 * (saturation to [-32768, 32767] or [-128, 127]).  shift = 0 saturates S
 * directly.
 *   A, B, b_layout, K limit and errors: as gemm_s8s8_s32.
 *   C: M x N row-major int16 / int8 (ldc >= N elements), fully overwritten
 *   in [0,M) x [0,N); any alignment.
 *   shift: 0 .. 31, else GEMM_ERR_INVALID_ARG.
 * Bit-exact: the result is a function of the exact sum only.
 */
gemm_status_t gemm_s8s8_s16(int64_t M, int64_t N, int64_t K,
                            const int8_t *A, int64_t lda,
                            const int8_t *B, int64_t ldb, int b_layout,
                            int16_t *C, int64_t ldc, int shift, gemm_stream_t stream);
gemm_status_t gemm_s8s8_s8(int64_t M, int64_t N, int64_t K,
                           const int8_t *A, int64_t lda,
                           const int8_t *B, int64_t ldb, int b_layout,
                           int8_t *C, int64_t ldc, int shift, gemm_stream_t stream);

/*
 * bf16-bf16 (Sec. 5.1, Table 1): C[i][j] = rne_bf16(sum_k a_ik * b_kj) with
 * the sum accumulated in float32 (any order) and rounded once to bf16,
 * nearest-even.  A, B, C are bf16 bit patterns (uint16_t).
 *   A: M x K row-major (lda >= K).  B: layout per b_layout.
 *   C: M x N row-major (ldc >= N), fully overwritten in [0,M) x [0,N).
 * Accuracy contract: |C - ref| <= 2^-8 |ref| + 2^-20 sum_k |a_ik b_kj| per
 * element, ref being the exact sum.
 */
gemm_status_t gemm_bf16_f32acc_bf16(int64_t M, int64_t N, int64_t K,
                                    const uint16_t *A, int64_t lda,
                                    const uint16_t *B, int64_t ldb, int b_layout,
                                    uint16_t *C, int64_t ldc, gemm_stream_t stream);

/*
 * Size of the fixed device scratch array used by gemm_s8s8_s32_noalloc.
 * A GPU holds this much memory from the first gemm_s8s8_s32_noalloc call on
 * it (which loads the array) until the process exits.
 */
#define GEMM_NOALLOC_SCRATCH_BYTES ((size_t)128 << 20) /* 128 MiB */

/*
 * gemm_s8s8_s32_noalloc -- the same exact int8 GEMM as gemm_s8s8_s32, for
 * callers that cannot let the library allocate device memory: an
 * application whose own allocator holds nearly all device memory, a service
 * enforcing a hard memory budget through its own allocator, or a
 * latency-critical loop that cannot afford cudaMalloc/cudaFree and their
 * synchronisation.  (The paper has no counterpart: it is an interface
 * convenience of this library.)
 *
 *   Arguments, layouts, results and errors are those of gemm_s8s8_s32, and
 *   the caller still owns A, B and C.  The results are those of
 *   gemm_s8s8_s32 bit for bit, but not always its speed: this entry point
 *   always stages both operands and runs the general tensor-core kernels,
 *   never the CUDA-core kernel for very small M or the kernel that converts
 *   a large operand in place.  The operands' bf16 staging copies and
 *   any split-K partial sums live in one static device array of
 *   GEMM_NOALLOC_SCRATCH_BYTES bytes instead of the library's workspace; the
 *   call never calls cudaMalloc, cudaFree or any other allocating routine.
 *   Bytes needed: round256(2*M*K8) + round256(2*K8*N) for column-major B
 *   (round256(2*M*K8) + round256(2*K*N8) for row-major B), plus
 *   round256(4*S*M*N) when the planner splits K into S > 1 parts (S <= 16,
 *   only for problems with fewer output tiles than SMs, unless
 *   GB300_GEMM_SPLITS overrides the planner), where K8 and N8 are
 *   K and N rounded up to multiples of 8.  A problem needing more returns
 *   GEMM_ERR_UNSUPPORTED and launches nothing.
 *
 *   The first call on each device loads the array -- that is the moment the
 *   GPU gives up its GEMM_NOALLOC_SCRATCH_BYTES -- and looks up its device
 *   address (cudaGetSymbolAddress) with that device current, then caches it.
 *   So make that first call (any valid problem will do) before the caller's
 *   own allocator reserves the device's memory, and before any stream
 *   capture.  After a cudaDeviceReset() call gemm_release_resources(), which
 *   forgets the cached address, before the next call.  All calls share the one array and
 *   it keeps whatever the last call left in it; every byte a call reads from
 *   it is written earlier in the same call, so nothing needs clearing.  Calls
 *   whose execution overlaps on the GPU (on different streams, or from
 *   several host threads) race on the array and corrupt each other's
 *   results: order them on one stream or synchronise between them.
 */
gemm_status_t gemm_s8s8_s32_noalloc(int64_t M, int64_t N, int64_t K,
                                    const int8_t *A, int64_t lda,
                                    const int8_t *B, int64_t ldb, int b_layout,
                                    int32_t *C, int64_t ldc, gemm_stream_t stream);

/* Human-readable name of a status code (static string, never NULL). */
const char *gemm_status_string(gemm_status_t status);

/*
 * Reads and clears the device error word that kernels set when a bounded
 * wait expires (GEMM_ERR_TIMEOUT) on the current device.  Synchronises the
 * device first.  Returns GEMM_OK if no kernel reported an error.
 */
gemm_status_t gemm_device_status(void);

/* Frees the workspace and cached state (device addresses looked up at the
 * first call, including the no-allocation scratch's) of the current device.
 * The caller must ensure no library kernel is still running.  Call it after
 * a cudaDeviceReset() before using the library on that device again. */
void gemm_release_resources(void);

/* Number of kernel launches the library has enqueued since load (all
 * devices); lets a caller count the kernels a region of work launched. */
uint64_t gemm_launch_count(void);

/* Re-reads the planner overrides (GB300_GEMM_BN ... GB300_GEMM_DEBUG, listed
 * at the top of this file) from the environment; otherwise they are read
 * once, at the first GEMM call.  A test and benchmark aid (the paper has no
 * counterpart); calls already enqueued are not affected. */
void gemm_reload_overrides(void);

/*
 * Failure-detection self-test (a diagnostic; the paper has no counterpart).
 * Launches one thread that waits, with the same bounded mbarrier wait the
 * GEMM kernels use, on a barrier nothing arrives on.  After `limit_ns`
 * (1 .. 1e9 ns, else GEMM_ERR_INVALID_ARG) the wait gives up and records
 * GEMM_ERR_TIMEOUT in the device error word; gemm_device_status() then
 * reports (and clears) it.  The kernel ends normally and the context stays
 * usable.  Returns GEMM_OK once the probe is launched.
 */
gemm_status_t gemm_selftest_wait_timeout(uint64_t limit_ns, gemm_stream_t stream);

/*
 * The plan the library would use for a GEMM (a host-only query: no device
 * is touched, so it also runs on a machine without a GPU).  The planner is
 * the GB300 restatement of the paper's tile model and balanced-point search
 * (Sec. 4.5.1 Eq. 1-5, Sec. 4.5.2 Eq. 6-10): among the compiled kernel
 * variants -- one CTA per 128 x BN tile or a CTA pair per 256 x BN tile --
 * and K splits it takes the least modelled time, from per-variant costs
 * fitted to measurements on GB300.
 *   int8: nonzero for the int8 entry points, 0 for bf16.  b_layout as in
 *   the GEMM calls.  sms: SMs of the device (152 on GB300); pair_slots:
 *   co-resident CTA pairs (76).  Operands are taken as tight (lda = K, ldb
 *   and ldc = N or K) and 16-byte aligned; the planner overrides in force
 *   (GB300_GEMM_*) apply.
 *   out->route: GEMM_ROUTE_*; bn: tile width (the small operand's tile
 *   height for GEMM_ROUTE_SMALL_OPERAND); splits: K split factor;
 *   tail_splits: 0, or the split of the tiles of the last, partly filled
 *   round of the tensor-core kernel (each in tail_splits K ranges, summed
 *   by the split-K reduction over those tiles only); stages:
 *   pipeline depth of the tensor-core kernel; grid: CTAs launched;
 *   model_us: modelled time of the tensor-core kernel and split-K reduction
 *   (the quantity the planner minimises); dram_us: the DRAM time of the
 *   model's traffic at the copy bandwidth (above model_us: memory-bound).
 * Returns GEMM_ERR_INVALID_ARG / GEMM_ERR_UNSUPPORTED like the GEMM calls.
 */
enum {
  GEMM_ROUTE_NONE = 0,           /* M == 0 or N == 0: nothing to do */
  GEMM_ROUTE_ZERO_FILL = 1,      /* K == 0 */
  GEMM_ROUTE_SMALL_M = 2,        /* CUDA-core kernel for very small M */
  GEMM_ROUTE_SMALL_OPERAND = 3,  /* int8 with one operand of <= 128 rows, converted in the kernel */
  GEMM_ROUTE_TC_SINGLE = 4,      /* tensor-core kernel, one CTA per 128 x BN tile */
  GEMM_ROUTE_TC_PAIR = 5,        /* tensor-core kernel, a CTA pair per 256 x BN tile */
  GEMM_ROUTE_TINY = 6            /* int8 problem small enough for one CUDA-core launch */
};
typedef struct {
  int route;
  int bn;
  int splits;
  int stages;
  int grid;
  double model_us;
  double dram_us;
  int tail_splits;
} gemm_plan_t;
gemm_status_t gemm_plan_query(int64_t M, int64_t N, int64_t K, int int8, int b_layout, int sms, int pair_slots,
                              gemm_plan_t *out);

/*
 * Read-bandwidth diagnostic (the paper has no counterpart): enqueues one
 * kernel that reads `bytes` of device memory at `ptr` with 16-byte loads
 * (four blocks per SM, several loads in flight per thread) and discards
 * them, so that the time between two events around it is what a plain read
 * of that many bytes takes -- the ceiling an HBM-bound GEMM of the same
 * traffic could reach.  ptr 16-byte aligned, bytes a multiple of 16, else
 * GEMM_ERR_INVALID_ARG.  Nothing is written to `ptr`'s buffer.
 */
gemm_status_t gemm_selftest_read_stream(const void *ptr, size_t bytes, gemm_stream_t stream);

/*
 * Profiling aid.  With both arguments non-NULL (cudaEvent_t handles created
 * by the caller), every following GEMM call records `start_event` on its
 * stream just before launching its main kernel (the tensor-core kernel, or
 * the CUDA-core kernel for very small M) and `stop_event` just after, so the
 * time between them covers that kernel alone -- not the operand staging or
 * split-K reduction passes.  Pass NULL, NULL to stop.  Process-wide setting;
 * not meant for concurrent callers.
 */
void gemm_profile_events(void *start_event, void *stop_event);

#if defined(__GNUC__)
#pragma GCC visibility pop
#endif
#ifdef __cplusplus
}
#endif

#endif /* GB300_GEMM_H */

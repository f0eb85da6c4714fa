/*
 * CPU oracle for the dense GEMM C = A.B -- TEST INFRASTRUCTURE ONLY.
 *
 * This file is the plain, slow, obviously correct statement of what the GPU
 * library computes.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it.  It shares no code, header or constant with
 * the CUDA library, and the CUDA library never loads it.
 *
 * What it follows in the paper ("Striking the Balance: GEMM Performance
 * Optimization Across Generations of Ryzen AI NPUs", arXiv 2512.13282):
 *   - Sec. 4.1: the problem is an M x K by K x N product giving C (M x N);
 *     A holds activations, B weights.
 *   - Sec. 4.2.2: A and C are row-major; B is row-major (K x N) or
 *     column-major (stored as N x K).
 *   - Sec. 5.1 / Table 1: the precisions "int8-int32" (int8 operands, full
 *     int32 output) and "bf16-bf16" (bf16 operands, bf16 output).
 *   - Sec. 4.2.1: K is reduced in time into a stationary accumulator that
 *     starts at zero; the order of that reduction is not fixed by the paper.
 *
 * The paper states neither the accumulation precision of bf16 nor a rounding
 * mode, nor what happens when int32 overflows.  The readings taken here are:
 *   - int8:  C[i][j] = sum_k A[i][k]*B(k,j) computed exactly in int64; the
 *            caller checks that it fits int32 (it always does for K <= 131071).
 *   - int8 reduced-precision outputs (Sec. 5.1 mentions int8-int16 and
 *            int8-int8 "precision reduction" without a rule): the exact sum
 *            divided by 2^shift, rounded to nearest with ties to even, then
 *            saturated to the output's range (oracle_requantize).
 *   - bf16:  inputs decoded exactly to double; ref = sum_k a*b and
 *            mag = sum_k |a*b| in double (every product is exact in double);
 *            rne_bf16() rounds a double straight to the nearest bf16, ties to
 *            even, with no intermediate float rounding.
 *
 * Loop order is the plain one: rows i (OpenMP-parallel), then k, then j, as
 * a row of C accumulates.  No blocking, no reordering.
 *
 * Parity pins: every function here is checked by the CPU tests against hand
 * cases, closed forms (all -128 inputs, identity and permutation matrices),
 * linearity in B and in A, layout equivalence, integer-valued bf16 inputs
 * whose sums are exact in float, and library conversions (torch float ->
 * bfloat16) for the rounding routine.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* B-layout flag values (Sec. 4.2.2): 0 = row-major K x N, 1 = column-major,
 * i.e. stored N x K with K contiguous. */
#define ORACLE_B_ROW_MAJOR 0
#define ORACLE_B_COL_MAJOR 1

/* Element (k, j) of the logical K x N matrix B, whatever its storage. */
static inline int64_t b_index(int64_t k, int64_t j, int64_t ldb, int layout) {
  return layout == ORACLE_B_ROW_MAJOR ? k * ldb + j : j * ldb + k;
}

/* bf16 bits -> double.  A bf16 value is the upper half of an IEEE binary32,
 * so the conversion is exact: shift into a float, widen to double. */
static inline double bf16_to_double(uint16_t bits) {
  uint32_t w = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &w, sizeof f);
  return (double)f;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

static int check_args(int64_t M, int64_t N, int64_t K, int64_t lda, int64_t ldb,
                      int layout, int64_t ldc) {
  if (M < 0 || N < 0 || K < 0) return 1;
  if (layout != ORACLE_B_ROW_MAJOR && layout != ORACLE_B_COL_MAJOR) return 1;
  if (K > 0 && M > 0 && lda < K) return 1;
  if (K > 0 && N > 0) {
    if (layout == ORACLE_B_ROW_MAJOR && ldb < N) return 1;
    if (layout == ORACLE_B_COL_MAJOR && ldb < K) return 1;
  }
  if (M > 0 && ldc < N) return 1;
  return 0;
}

/* int8-int32 path, exact: C (int64, M x N, leading dimension ldc). */
int oracle_gemm_s8(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                   const int8_t *B, int64_t ldb, int layout, int64_t *C, int64_t ldc) {
  if (check_args(M, N, K, lda, ldb, layout, ldc)) return 1;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t i = 0; i < M; ++i) {
    int64_t *c = C + i * ldc;
    for (int64_t j = 0; j < N; ++j) c[j] = 0;
    for (int64_t k = 0; k < K; ++k) {
      const int64_t a = A[i * lda + k];
      for (int64_t j = 0; j < N; ++j) c[j] += a * (int64_t)B[b_index(k, j, ldb, layout)];
    }
  }
  return 0;
}

/* bf16-bf16 path: ref = sum a*b and mag = sum |a*b|, both in double. */
int oracle_gemm_bf16(int64_t M, int64_t N, int64_t K, const uint16_t *A, int64_t lda,
                     const uint16_t *B, int64_t ldb, int layout, double *ref, double *mag,
                     int64_t ldc) {
  if (check_args(M, N, K, lda, ldb, layout, ldc)) return 1;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t i = 0; i < M; ++i) {
    double *r = ref + i * ldc;
    double *g = mag + i * ldc;
    for (int64_t j = 0; j < N; ++j) { r[j] = 0.0; g[j] = 0.0; }
    for (int64_t k = 0; k < K; ++k) {
      const double a = bf16_to_double(A[i * lda + k]);
      for (int64_t j = 0; j < N; ++j) {
        const double p = a * bf16_to_double(B[b_index(k, j, ldb, layout)]);
        r[j] += p;
        g[j] += fabs(p);
      }
    }
  }
  return 0;
}

/* Selected entries (rows[t], cols[t]) of the int8 product, one dot product
 * each; used where the full product is too large for the CPU. */
int oracle_gemm_s8_entries(int64_t M, int64_t N, int64_t K, const int8_t *A, int64_t lda,
                           const int8_t *B, int64_t ldb, int layout, const int64_t *rows,
                           const int64_t *cols, int64_t count, int64_t *out) {
  if (check_args(M, N, K, lda, ldb, layout, N)) return 1;
  for (int64_t t = 0; t < count; ++t)
    if (rows[t] < 0 || rows[t] >= M || cols[t] < 0 || cols[t] >= N) return 1;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < count; ++t) {
    const int64_t i = rows[t], j = cols[t];
    int64_t s = 0;
    for (int64_t k = 0; k < K; ++k)
      s += (int64_t)A[i * lda + k] * (int64_t)B[b_index(k, j, ldb, layout)];
    out[t] = s;
  }
  return 0;
}

int oracle_gemm_bf16_entries(int64_t M, int64_t N, int64_t K, const uint16_t *A, int64_t lda,
                             const uint16_t *B, int64_t ldb, int layout, const int64_t *rows,
                             const int64_t *cols, int64_t count, double *ref, double *mag) {
  if (check_args(M, N, K, lda, ldb, layout, N)) return 1;
  for (int64_t t = 0; t < count; ++t)
    if (rows[t] < 0 || rows[t] >= M || cols[t] < 0 || cols[t] >= N) return 1;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < count; ++t) {
    const int64_t i = rows[t], j = cols[t];
    double r = 0.0, g = 0.0;
    for (int64_t k = 0; k < K; ++k) {
      const double p = bf16_to_double(A[i * lda + k]) * bf16_to_double(B[b_index(k, j, ldb, layout)]);
      r += p;
      g += fabs(p);
    }
    ref[t] = r;
    mag[t] = g;
  }
  return 0;
}

/* Round a double to the nearest bf16, ties to even (the output rounding the
 * bf16 path is held to).  bf16 has an 8-bit significand and the binary32
 * exponent range: normals from 2^-126, subnormals in steps of 2^-133, the
 * largest finite value (2 - 2^-7) * 2^127.
 *
 * For |x| in [2^E, 2^(E+1)) (E clamped below at -126, where the spacing stops
 * shrinking) the spacing of bf16 values is q = 2^(E-7).  m = |x|/q is exact
 * (a power-of-two scaling) and lies in [128, 256) (or below 128 in the
 * subnormal range); rint() rounds it to an integer r, ties to even, under the
 * default rounding mode.  The encoding is then ((E + 127) << 7) + r - 128: a
 * carry to r = 256 moves to the next binade with a zero fraction, and at
 * E = 127 that gives 0x7F80, infinity; at E = -126 with r < 128 it gives the
 * subnormal fraction r. */
static uint16_t rne_bf16_one(double x) {
  const uint16_t sign = signbit(x) ? 0x8000u : 0u;
  if (isnan(x)) return (uint16_t)(sign | 0x7FC0u);
  const double ax = fabs(x);
  if (isinf(ax)) return (uint16_t)(sign | 0x7F80u);
  if (ax == 0.0) return sign;
  int e;
  (void)frexp(ax, &e);      /* ax = f * 2^e with f in [0.5, 1) */
  int E = e - 1;            /* ax in [2^E, 2^(E+1)) */
  if (E > 127) return (uint16_t)(sign | 0x7F80u);
  if (E < -126) E = -126;
  const double r = rint(ldexp(ax, 7 - E));
  const long enc = ((long)(E + 127) << 7) + (long)r - 128;
  return (uint16_t)(sign | (uint16_t)enc);
}

void oracle_rne_bf16(const double *x, uint16_t *out, int64_t n) {
  for (int64_t t = 0; t < n; ++t) out[t] = rne_bf16_one(x[t]);
}

/* Reduced-precision int8 outputs: acc / 2^shift rounded to nearest (ties to
 * even), saturated to [-2^(bits-1), 2^(bits-1) - 1].  shift in [0, 62],
 * bits in {8, 16, 32}.  Floor division is written out (no shift of negative
 * numbers): q = floor(acc / 2^shift), r = acc - q * 2^shift in [0, 2^shift). */
int oracle_requantize(const int64_t *acc, int64_t n, int shift, int bits, int64_t *out) {
  if (shift < 0 || shift > 62 || (bits != 8 && bits != 16 && bits != 32)) return 1;
  const int64_t d = (int64_t)1 << shift;
  const int64_t hi = ((int64_t)1 << (bits - 1)) - 1, lo = -((int64_t)1 << (bits - 1));
  for (int64_t t = 0; t < n; ++t) {
    const int64_t a = acc[t];
    int64_t q = a / d;               /* truncates toward zero */
    if (a % d != 0 && a < 0) q -= 1; /* floor */
    const int64_t r = a - q * d;     /* 0 <= r < d */
    if (shift > 0) {
      const int64_t half = d / 2;
      if (r > half || (r == half && (q % 2 != 0))) q += 1;
    }
    out[t] = q > hi ? hi : (q < lo ? lo : q);
  }
  return 0;
}

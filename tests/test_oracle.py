"""Pins for the CPU oracle (no GPU).

The oracle is only trusted because these checks tie it to something other
than itself: hand-worked products, closed forms, invariants, library routines
on special cases, and brute force on tiny inputs.  Each check is a ``pin_*``
function taking an oracle library handle, so that ``test_mutants_are_caught``
can rebuild the oracle with a planted mistake (a dropped term, a wrong sign,
a transposed operand, a broken rounding) and show that some pin fails.
"""
import os
import re
import shutil

import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import workloads as W
from tests import golden_cases

ROW, COL = oracle.B_ROW_MAJOR, oracle.B_COL_MAJOR


def _to_col(B_row: np.ndarray) -> np.ndarray:
    """Column-major storage (N x K) of a row-major K x N matrix."""
    return np.ascontiguousarray(B_row.T)


def _bf16_from_f32(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16) \
        .view(torch.int16).numpy().view(np.uint16)


def _decode_torch(bits: np.ndarray) -> np.ndarray:
    """Library decode of bf16 bits (torch bfloat16 -> float64)."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16) \
        .to(torch.float64).numpy()


# ---------------------------------------------------------------- pins ----

def pin_golden(lib):
    """Hand-worked products (tests/golden/hand_cases.txt)."""
    for c in golden_cases.load():
        if c["dtype"] == "int8":
            got = oracle.gemm_s8(c["A"], c["B"], c["layout"], lib=lib)
            assert np.array_equal(got, c["C"].astype(np.int64)), c["name"]
        else:
            ref, mag = oracle.gemm_bf16(c["A"], c["B"], c["layout"], lib=lib)
            assert np.array_equal(ref, c["C"]), c["name"]
            assert np.array_equal(mag, c["MAG"]), c["name"]
            assert np.array_equal(oracle.rne_bf16(ref, lib=lib), c["RNE"]), c["name"]


def pin_k0_k1(lib):
    """K = 0 gives zeros; K = 1 is the outer product (numpy.outer)."""
    A = W.random_int8((5, 0), 1)
    B = W.random_int8((0, 7), 2)
    assert np.array_equal(oracle.gemm_s8(A, B, ROW, lib=lib), np.zeros((5, 7), np.int64))
    a = W.random_int8((6, 1), 3)
    b = W.random_int8((1, 4), 4)
    outer = np.outer(a[:, 0].astype(np.int64), b[0].astype(np.int64))
    assert np.array_equal(oracle.gemm_s8(a, b, ROW, lib=lib), outer)
    assert np.array_equal(oracle.gemm_s8(a, _to_col(b), COL, lib=lib), outer)
    fa, fb = W.random_bf16((6, 1), 5), W.random_bf16((1, 4), 6)
    ref, mag = oracle.gemm_bf16(fa, fb, ROW, lib=lib)
    o = np.outer(_decode_torch(fa)[:, 0], _decode_torch(fb)[0])
    assert np.array_equal(ref, o) and np.array_equal(mag, np.abs(o))


def pin_dot_closed_forms(lib):
    """M = N = 1: a ones row times B sums B's column; alternating signs give
    the alternating sum."""
    K = 1001
    b = W.random_int8((K, 1), 7)
    ones = np.ones((1, K), np.int8)
    assert oracle.gemm_s8(ones, b, ROW, lib=lib)[0, 0] == int(b.astype(np.int64).sum())
    alt = np.where(np.arange(K) % 2 == 0, 1, -1).astype(np.int8)[None, :]
    want = int(b[0::2].astype(np.int64).sum() - b[1::2].astype(np.int64).sum())
    assert oracle.gemm_s8(alt, b, ROW, lib=lib)[0, 0] == want


def pin_identity_permutation(lib):
    """A.I = A, I.B = B, A.P permutes columns, P.B permutes rows (both B layouts)."""
    rng = np.random.default_rng(11)
    M, K, N = 9, 13, 11
    A = W.random_int8((M, K), 8)
    B = W.random_int8((K, N), 9)
    I_k = np.eye(K, dtype=np.int8)
    for lay, Bs in ((ROW, I_k), (COL, _to_col(I_k))):
        assert np.array_equal(oracle.gemm_s8(A, Bs, lay, lib=lib), A.astype(np.int64))
    assert np.array_equal(oracle.gemm_s8(np.eye(K, dtype=np.int8), B, ROW, lib=lib), B.astype(np.int64))
    perm = rng.permutation(K)
    P = np.zeros((K, K), np.int8)
    P[perm, np.arange(K)] = 1            # (A.P)[:, j] = A[:, perm[j]]
    for lay, Ps in ((ROW, P), (COL, _to_col(P))):
        assert np.array_equal(oracle.gemm_s8(A, Ps, lay, lib=lib), A[:, perm].astype(np.int64))
    Q = np.zeros((K, K), np.int8)
    Q[np.arange(K), perm] = 1            # (Q.B)[i, :] = B[perm[i], :]
    assert np.array_equal(oracle.gemm_s8(Q, B, ROW, lib=lib), B[perm].astype(np.int64))
    Bf = W.random_bf16((K, N), 10)
    If = _bf16_from_f32(np.eye(K))
    ref, mag = oracle.gemm_bf16(If, Bf, ROW, lib=lib)
    assert np.array_equal(ref, _decode_torch(Bf)) and np.array_equal(mag, np.abs(_decode_torch(Bf)))


def pin_extremes(lib):
    """All -128 gives 16384*K; -128 x 127 gives -16256*K; K = 131071 all -128
    is 2147467264 (fits int32); K = 131072 is 2^31 (does not)."""
    for K, N in ((1, 3), (64, 5), (1024, 2), (4097, 3)):
        A = np.full((3, K), -128, np.int8)
        B = np.full((K, N), -128, np.int8)
        assert (oracle.gemm_s8(A, B, ROW, lib=lib) == 16384 * K).all()
        B2 = np.full((N, K), 127, np.int8)
        assert (oracle.gemm_s8(A, B2, COL, lib=lib) == -16256 * K).all()
    for K, want in ((131071, 2147467264), (131072, 2 ** 31)):
        A = np.full((1, K), -128, np.int8)
        B = np.full((K, 1), -128, np.int8)
        assert oracle.gemm_s8_entries(A, B, ROW, [0], [0], lib=lib)[0] == want


def pin_linearity(lib):
    """C(A, B1+B2) = C(A, B1) + C(A, B2) and C(A1+A2, B) = C(A1, B) + C(A2, B)
    with entries in [-64, 63] so the sums stay int8."""
    M, K, N = 7, 37, 10
    A = W.random_int8((M, K), 12)
    B1, B2 = W.random_int8((K, N), 13, -64, 63), W.random_int8((K, N), 14, -64, 63)
    for lay, f in ((ROW, lambda x: x), (COL, _to_col)):
        lhs = oracle.gemm_s8(A, f(B1 + B2), lay, lib=lib)
        rhs = oracle.gemm_s8(A, f(B1), lay, lib=lib) + oracle.gemm_s8(A, f(B2), lay, lib=lib)
        assert np.array_equal(lhs, rhs)
    A1, A2 = W.random_int8((M, K), 15, -64, 63), W.random_int8((M, K), 16, -64, 63)
    B = W.random_int8((K, N), 17)
    assert np.array_equal(oracle.gemm_s8(A1 + A2, B, ROW, lib=lib),
                          oracle.gemm_s8(A1, B, ROW, lib=lib) + oracle.gemm_s8(A2, B, ROW, lib=lib))


def pin_layout_and_transpose(lib):
    """Column-major B equals its row-major copy, bit for bit, on both paths;
    (A.B)^T = B^T.A^T."""
    M, K, N = 6, 19, 8
    A, B = W.random_int8((M, K), 18), W.random_int8((K, N), 19)
    C = oracle.gemm_s8(A, B, ROW, lib=lib)
    assert np.array_equal(C, oracle.gemm_s8(A, _to_col(B), COL, lib=lib))
    Ct = oracle.gemm_s8(np.ascontiguousarray(B.T), np.ascontiguousarray(A.T), ROW, lib=lib)
    assert np.array_equal(C.T, Ct)
    Af, Bf = W.random_bf16((M, K), 20), W.random_bf16((K, N), 21)
    r1, m1 = oracle.gemm_bf16(Af, Bf, ROW, lib=lib)
    r2, m2 = oracle.gemm_bf16(Af, _to_col(Bf), COL, lib=lib)
    assert np.array_equal(r1, r2) and np.array_equal(m1, m2)


def pin_numpy_int(lib):
    """Brute force on small inputs against numpy's exact int64 matmul, with
    ragged sizes and leading dimensions wider than the rows."""
    for (M, K, N, seed) in ((1, 1, 1, 30), (3, 5, 2, 31), (17, 33, 9, 32), (40, 70, 23, 33)):
        A_full = W.random_int8((M, K + 3), seed)
        A = A_full[:, :K]
        B = W.random_int8((K, N), seed + 100)
        want = A.astype(np.int64) @ B.astype(np.int64)
        assert np.array_equal(oracle.gemm_s8(A, B, ROW, lib=lib), want)
        Bc_full = W.random_int8((N, K + 5), seed + 200)
        Bc = Bc_full[:, :K]
        want_c = A.astype(np.int64) @ Bc.astype(np.int64).T
        assert np.array_equal(oracle.gemm_s8(A, Bc, COL, lib=lib), want_c)


def pin_numpy_float(lib):
    """bf16 path against numpy float64 matmul of library-decoded inputs:
    ref within float64 rounding of A@B, mag equal to |A|@|B| to rounding."""
    for (M, K, N, seed) in ((4, 9, 3, 40), (16, 64, 12, 41), (9, 300, 5, 42)):
        A, B = W.random_bf16((M, K), seed), W.random_bf16((K, N), seed + 1)
        a, b = _decode_torch(A), _decode_torch(B)
        ref, mag = oracle.gemm_bf16(A, B, ROW, lib=lib)
        want_mag = np.abs(a) @ np.abs(b)
        assert np.allclose(mag, want_mag, rtol=1e-13, atol=0)
        assert (np.abs(ref - a @ b) <= 1e-13 * want_mag).all()


def pin_integer_bf16_exact(lib):
    """Integer-valued bf16 inputs in [-8, 8]: every partial sum is an integer
    below 2^24, so float32 accumulation (torch) is exact and the bf16 rounding
    of it must equal the oracle's rne_bf16(ref) bit for bit."""
    M, K, N = 12, 300, 9
    A, B = W.integer_bf16((M, K), 50), W.integer_bf16((K, N), 51)
    ref, _ = oracle.gemm_bf16(A, B, ROW, lib=lib)
    a = torch.from_numpy(_decode_torch(A)).to(torch.float32)
    b = torch.from_numpy(_decode_torch(B)).to(torch.float32)
    want = (a @ b).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ref, (a @ b).to(torch.float64).numpy())
    assert np.array_equal(oracle.rne_bf16(ref, lib=lib), want)


def pin_rne_vs_torch(lib):
    """rne_bf16 on float32-representable values equals torch's float32 ->
    bfloat16 conversion (round to nearest even): random bit patterns over the
    whole exponent range, subnormals, exact ties, the overflow boundary."""
    rng = np.random.default_rng(60)
    bits = rng.integers(0, 2 ** 32, size=200000, dtype=np.uint64).astype(np.uint32)
    f = bits.view(np.float32)
    f = f[np.isfinite(f)]
    ties = ((rng.integers(0, 2 ** 16, 5000).astype(np.uint32) << 16) | 0x8000).view(np.float32)
    ties = ties[np.isfinite(ties)]
    special = np.array([0.0, -0.0, 1.0, -1.0, 2.0 ** -126, 2.0 ** -133, 2.0 ** -134, 3 * 2.0 ** -135,
                        3.3895313892515355e38, 3.39e38, 3.3961e38, 3.3963e38,
                        float(np.finfo(np.float32).max), 1e-40, -1e-40], dtype=np.float32)
    for x in (f, ties, special):
        want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        got = oracle.rne_bf16(x.astype(np.float64), lib=lib)
        assert np.array_equal(got, want)


def pin_rne_double_cases(lib):
    """Cases a float32 detour would get wrong, and specials, worked by hand:
    1 + 2^-8 is a tie (to even: 1.0, 0x3f80); 1 + 2^-8 + 2^-40 is above the
    tie (0x3f81); 2^128 overflows to +inf (0x7f80); NaN stays NaN."""
    x = np.array([1 + 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -40, -(1 + 2.0 ** -8 + 2.0 ** -40),
                  1 + 3 * 2.0 ** -8, 2.0 ** 128, -np.inf, 1e300, 1e-300, -1e-300])
    want = np.array([0x3F80, 0x3F81, 0xBF81, 0x3F82, 0x7F80, 0xFF80, 0x7F80, 0x0000, 0x8000], np.uint16)
    assert np.array_equal(oracle.rne_bf16(x, lib=lib), want)
    nan = oracle.rne_bf16(np.array([np.nan]), lib=lib)[0]
    assert (nan & 0x7F80) == 0x7F80 and (nan & 0x007F) != 0


def pin_entries(lib):
    """The selected-entries routines agree with the full products."""
    M, K, N = 21, 45, 17
    A, B = W.random_int8((M, K), 70), W.random_int8((N, K), 71)
    C = oracle.gemm_s8(A, B, COL, lib=lib)
    rows, cols = np.arange(M * N) // N, np.arange(M * N) % N
    assert np.array_equal(oracle.gemm_s8_entries(A, B, COL, rows, cols, lib=lib), C.ravel())
    Af, Bf = W.random_bf16((M, K), 72), W.random_bf16((K, N), 73)
    ref, mag = oracle.gemm_bf16(Af, Bf, ROW, lib=lib)
    r, g = oracle.gemm_bf16_entries(Af, Bf, ROW, rows, cols, lib=lib)
    assert np.array_equal(r, ref.ravel()) and np.array_equal(g, mag.ravel())


def pin_requantize(lib):
    """Shift-round-saturate: hand-worked ties (to even) and saturation, and
    numpy's round-half-even division plus clipping on random sums."""
    acc = np.array([5, 7, -5, -7, 6, -6, 1, -1, 3, -3, 0, 40000, -40000, 2**31 - 1, -2**31], np.int64)
    want1 = np.array([2, 4, -2, -4, 3, -3, 0, 0, 2, -2, 0, 20000, -20000, 2**30, -2**30], np.int64)
    assert np.array_equal(oracle.requantize(acc, 1, 32, lib=lib), want1)
    assert np.array_equal(oracle.requantize(acc, 0, 16, lib=lib),
                          np.clip(acc, -32768, 32767))
    assert np.array_equal(oracle.requantize(np.array([383, 384, 385, -383, -384, -385], np.int64), 8, 8, lib=lib),
                          np.array([1, 2, 2, -1, -2, -2], np.int64))  # 1.496, 1.5 -> 2 (even), 1.504
    rng = np.random.default_rng(90)
    a = rng.integers(-2**31, 2**31, 5000, dtype=np.int64)
    for shift, bits in ((3, 8), (7, 16), (13, 16), (20, 8), (31, 32)):
        want = np.clip(np.round(a / float(2 ** shift)), -(2 ** (bits - 1)), 2 ** (bits - 1) - 1).astype(np.int64)
        assert np.array_equal(oracle.requantize(a, shift, bits, lib=lib), want)


PINS = [pin_golden, pin_k0_k1, pin_dot_closed_forms, pin_identity_permutation, pin_extremes,
        pin_linearity, pin_layout_and_transpose, pin_numpy_int, pin_numpy_float,
        pin_integer_bf16_exact, pin_rne_vs_torch, pin_rne_double_cases, pin_entries, pin_requantize]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(None)


def test_argument_errors():
    A, B = W.random_int8((3, 4), 1), W.random_int8((5, 2), 2)
    with pytest.raises(ValueError):
        oracle.gemm_s8(A, B, ROW)
    with pytest.raises(ValueError):
        oracle.gemm_s8(A, W.random_int8((4, 2), 3), 7)
    with pytest.raises(ValueError):
        oracle.gemm_s8_entries(A, W.random_int8((4, 2), 3), ROW, [3], [0])


def test_bound_checker():
    """The bf16 acceptance rule: exact rounding passes; an error of 2^-7
    relative on a value with small mag fails; NaN matches NaN only."""
    ref = np.array([1.0, -3.0, 0.0, np.nan, np.inf])
    mag = np.array([1.0, 3.0, 0.0, np.nan, np.inf])
    good = oracle.rne_bf16(ref)
    assert oracle.bf16_within_bound(good, ref, mag).all()
    bad = oracle.rne_bf16(np.array([1.0 + 2.0 ** -6, -3.0 * (1 + 2.0 ** -6), 2.0 ** -10, 1.0, -np.inf]))
    assert not oracle.bf16_within_bound(bad, ref, mag).any()


# A plausible mistake anywhere in the oracle must fail at least one pin.
MUTANTS = {
    "dropped_last_term_s8": ("for (int64_t k = 0; k < K; ++k) {\n      const int64_t a",
                             "for (int64_t k = 0; k + 1 < K; ++k) {\n      const int64_t a"),
    "dropped_first_term_bf16": ("for (int64_t k = 0; k < K; ++k) {\n      const double a",
                                "for (int64_t k = 1; k < K; ++k) {\n      const double a"),
    "transposed_b": ("return layout == ORACLE_B_ROW_MAJOR ? k * ldb + j : j * ldb + k;",
                     "return layout == ORACLE_B_ROW_MAJOR ? k * ldb + j : k * ldb + j;"),
    "wrong_sign_s8": ("c[j] += a * (int64_t)B", "c[j] -= a * (int64_t)B"),
    "mag_not_abs": ("g[j] += fabs(p);", "g[j] += p;"),
    "lda_ignored": ("const int64_t a = A[i * lda + k];", "const int64_t a = A[i * K + k];"),
    "rne_truncates": ("const double r = rint(ldexp(ax, 7 - E));",
                      "const double r = floor(ldexp(ax, 7 - E));"),
    "rne_ties_away": ("const double r = rint(ldexp(ax, 7 - E));",
                      "const double r = round(ldexp(ax, 7 - E));"),
    "rne_no_subnormal_clamp": ("if (E < -126) E = -126;", ""),
    "requant_ties_away": ("if (r > half || (r == half && (q % 2 != 0))) q += 1;",
                          "if (r >= half) q += 1;"),
    "requant_no_floor": ("if (a % d != 0 && a < 0) q -= 1; /* floor */", ""),
    "entries_wrong_index": ("s += (int64_t)A[i * lda + k] * (int64_t)B[b_index(k, j, ldb, layout)];",
                            "s += (int64_t)A[j * lda + k] * (int64_t)B[b_index(k, i, ldb, layout)];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutants_are_caught(name, tmp_path):
    src = open(oracle._SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) == 1, f"mutation site for {name} not found"
    mpath = tmp_path / "mutant.c"
    mpath.write_text(src.replace(old, new))
    lib = oracle.open_lib(oracle.compile_c(str(mpath), str(tmp_path / "libmutant.so")))
    failures = 0
    for pin in PINS:
        try:
            pin(lib)
        except (AssertionError, ValueError):
            failures += 1
    assert failures > 0, f"mutant {name} passed every pin"

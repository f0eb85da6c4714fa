"""CPU oracle for C = A.B -- test infrastructure only.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg (``bench.py`` ``cpu_baseline`` and ``--impl reference``) may import this
package.  The CUDA library never loads it, and it loads nothing from the CUDA
library: the two share no code.

The arithmetic lives in ``oracle_gemm.c`` (plain C, OpenMP over rows); this
module only compiles it with gcc and marshals numpy arrays.  Paper passages
followed: Sec. 4.1 (the M x K by K x N product), Sec. 4.2.2 (A and C
row-major, B row-major K x N or column-major N x K), Sec. 5.1 / Table 1 (the
int8-int32 and bf16-bf16 precisions).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle_gemm.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

B_ROW_MAJOR = 0  # B stored K x N, row-major
B_COL_MAJOR = 1  # B stored N x K (column-major K x N)

_i64 = ctypes.c_int64
_ptr = ctypes.c_void_p


def compile_c(src: str, out: str) -> str:
    """gcc -O2 with OpenMP; no fast-math and no contraction, so every
    floating-point operation is the one written in the source."""
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` next to its source."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    return compile_c(_SRC, _LIB_PATH)


def open_lib(path: str):
    """Load a compiled oracle library and declare its C signatures."""
    lib = ctypes.CDLL(path)
    _declare(lib)
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        _lib = open_lib(build())
        return _lib


def _declare(lib):
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_gemm_s8.argtypes = [_i64, _i64, _i64, _ptr, _i64, _ptr, _i64, ctypes.c_int, _ptr, _i64]
    lib.oracle_gemm_bf16.argtypes = [_i64, _i64, _i64, _ptr, _i64, _ptr, _i64, ctypes.c_int, _ptr, _ptr, _i64]
    lib.oracle_gemm_s8_entries.argtypes = [_i64, _i64, _i64, _ptr, _i64, _ptr, _i64, ctypes.c_int,
                                           _ptr, _ptr, _i64, _ptr]
    lib.oracle_gemm_bf16_entries.argtypes = [_i64, _i64, _i64, _ptr, _i64, _ptr, _i64, ctypes.c_int,
                                             _ptr, _ptr, _i64, _ptr, _ptr]
    lib.oracle_rne_bf16.argtypes = [_ptr, _ptr, _i64]
    lib.oracle_requantize.argtypes = [_ptr, _i64, ctypes.c_int, ctypes.c_int, _ptr]
    lib.oracle_requantize.restype = ctypes.c_int
    for f in (lib.oracle_gemm_s8, lib.oracle_gemm_bf16, lib.oracle_gemm_s8_entries,
              lib.oracle_gemm_bf16_entries):
        f.restype = ctypes.c_int
    lib.oracle_rne_bf16.restype = None


def num_threads(lib=None) -> int:
    return int((lib or _load()).oracle_num_threads())


def _addr(a: np.ndarray) -> int:
    return a.ctypes.data if a.size else 0


def _check_2d(x: np.ndarray, dtype) -> np.ndarray:
    if x.dtype != dtype or x.ndim != 2 or (x.size and x.shape[1] > 1 and x.strides[1] != x.itemsize):
        raise ValueError(f"expected a 2-D {np.dtype(dtype)} array with unit column stride")
    return x


def _ld(x: np.ndarray) -> int:
    if x.size == 0 or x.shape[0] == 1:
        return max(x.shape[1], 1)
    return x.strides[0] // x.itemsize


def _shape(A: np.ndarray, B: np.ndarray, layout: int):
    M, K = A.shape
    if layout == B_ROW_MAJOR:
        Kb, N = B.shape
    elif layout == B_COL_MAJOR:
        N, Kb = B.shape
    else:
        raise ValueError("layout must be 0 (row-major K x N) or 1 (column-major, N x K)")
    if Kb != K:
        raise ValueError(f"inner dimensions differ: A has K={K}, B has K={Kb}")
    return M, N, K


def gemm_s8(A: np.ndarray, B: np.ndarray, layout: int = B_ROW_MAJOR, lib=None) -> np.ndarray:
    """Exact int8 x int8 product as an int64 M x N array."""
    _check_2d(A, np.int8), _check_2d(B, np.int8)
    M, N, K = _shape(A, B, layout)
    C = np.zeros((M, N), dtype=np.int64)
    rc = (lib or _load()).oracle_gemm_s8(M, N, K, _addr(A), _ld(A), _addr(B), _ld(B), layout,
                               _addr(C), max(N, 1))
    if rc:
        raise ValueError("oracle_gemm_s8 rejected its arguments")
    return C


def gemm_bf16(A: np.ndarray, B: np.ndarray, layout: int = B_ROW_MAJOR, lib=None):
    """bf16 product over bit patterns (uint16): returns (ref, mag) in float64,
    ref = sum a*b and mag = sum |a*b|."""
    _check_2d(A, np.uint16), _check_2d(B, np.uint16)
    M, N, K = _shape(A, B, layout)
    ref = np.zeros((M, N), dtype=np.float64)
    mag = np.zeros((M, N), dtype=np.float64)
    rc = (lib or _load()).oracle_gemm_bf16(M, N, K, _addr(A), _ld(A), _addr(B), _ld(B), layout,
                                 _addr(ref), _addr(mag), max(N, 1))
    if rc:
        raise ValueError("oracle_gemm_bf16 rejected its arguments")
    return ref, mag


def _entries_args(rows, cols):
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    cols = np.ascontiguousarray(cols, dtype=np.int64)
    if rows.shape != cols.shape or rows.ndim != 1:
        raise ValueError("rows and cols must be 1-D and the same length")
    return rows, cols


def gemm_s8_entries(A, B, layout, rows, cols, lib=None) -> np.ndarray:
    """Exact int8 product at the positions (rows[t], cols[t]) only."""
    _check_2d(A, np.int8), _check_2d(B, np.int8)
    M, N, K = _shape(A, B, layout)
    rows, cols = _entries_args(rows, cols)
    out = np.zeros(rows.shape, dtype=np.int64)
    rc = (lib or _load()).oracle_gemm_s8_entries(M, N, K, _addr(A), _ld(A), _addr(B), _ld(B), layout,
                                       _addr(rows), _addr(cols), rows.size, _addr(out))
    if rc:
        raise ValueError("oracle_gemm_s8_entries rejected its arguments")
    return out


def gemm_bf16_entries(A, B, layout, rows, cols, lib=None):
    """bf16 product (ref, mag) at the positions (rows[t], cols[t]) only."""
    _check_2d(A, np.uint16), _check_2d(B, np.uint16)
    M, N, K = _shape(A, B, layout)
    rows, cols = _entries_args(rows, cols)
    ref = np.zeros(rows.shape, dtype=np.float64)
    mag = np.zeros(rows.shape, dtype=np.float64)
    rc = (lib or _load()).oracle_gemm_bf16_entries(M, N, K, _addr(A), _ld(A), _addr(B), _ld(B), layout,
                                         _addr(rows), _addr(cols), rows.size, _addr(ref), _addr(mag))
    if rc:
        raise ValueError("oracle_gemm_bf16_entries rejected its arguments")
    return ref, mag


def rne_bf16(x, lib=None) -> np.ndarray:
    """Round float64 values straight to bf16 bit patterns (nearest, ties to even)."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.zeros(x.shape, dtype=np.uint16)
    (lib or _load()).oracle_rne_bf16(_addr(x), _addr(out), x.size)
    return out


def requantize(acc, shift: int, bits: int, lib=None) -> np.ndarray:
    """Reduced-precision int8 outputs: exact sums divided by 2^shift, rounded
    to nearest with ties to even, saturated to a signed `bits`-bit range."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    out = np.zeros(acc.shape, dtype=np.int64)
    if (lib or _load()).oracle_requantize(_addr(acc), acc.size, int(shift), int(bits), _addr(out)):
        raise ValueError("oracle_requantize: shift must be 0..62 and bits 8, 16 or 32")
    return out


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact decode of bf16 bit patterns (upper half of a binary32)."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def bf16_within_bound(C_bits, ref, mag):
    """Acceptance rule of the bf16 path, element by element:
    |C - ref| <= 2^-8 |ref| + 2^-20 mag, C decoded from bf16 and compared in
    float64.  NaN matches NaN; an infinity matches the same infinity.
    Returns a boolean array."""
    c = bf16_bits_to_f64(C_bits)
    ref = np.asarray(ref, dtype=np.float64)
    mag = np.asarray(mag, dtype=np.float64)
    with np.errstate(invalid="ignore", over="ignore"):
        ok = np.abs(c - ref) <= (2.0 ** -8) * np.abs(ref) + (2.0 ** -20) * mag
    ok &= np.isfinite(ref)
    both_nan = np.isnan(c) & np.isnan(ref)
    same_inf = np.isinf(c) & np.isinf(ref) & (np.sign(c) == np.sign(ref))
    # A finite ref whose allowed interval reaches past the bf16 overflow
    # threshold (2 - 2^-8) * 2^127 may round to the infinity of its sign.
    with np.errstate(invalid="ignore", over="ignore"):
        reach = np.abs(ref) * (1 + 2.0 ** -8) + (2.0 ** -20) * mag
        overflow = (np.isinf(c) & np.isfinite(ref) & (np.sign(c) == np.sign(ref))
                    & (reach >= (2 - 2.0 ** -8) * 2.0 ** 127))
    return ok | both_nan | same_inf | overflow

"""ctypes binding of the C ABI in ``include/gb300_gemm.h`` -- argument
marshalling only; every step of the GEMM runs in the library's CUDA kernels.

The functions keep the C names.  Pointer arguments accept either an integer
device address or a CUDA ``torch.Tensor`` (its ``data_ptr()``); ``stream``
accepts an integer ``cudaStream_t``, a ``torch.cuda.Stream`` or ``None``
(torch's current stream on the current device).

The library must have been built (``paper_2512_13282_gb300.build.build()``);
there is no fallback: loading fails loudly if it is missing.
"""
from __future__ import annotations

import ctypes
import os
import threading

from .build import LIB_PATH

GEMM_OK = 0
GEMM_ERR_INVALID_ARG = 1
GEMM_ERR_UNSUPPORTED = 2
GEMM_ERR_CUDA = 3
GEMM_ERR_TIMEOUT = 4

GEMM_NOALLOC_SCRATCH_BYTES = 128 << 20

GEMM_B_ROW_MAJOR_KxN = 0
GEMM_B_COL_MAJOR_NxK = 1

GEMM_ROUTE_NONE = 0
GEMM_ROUTE_ZERO_FILL = 1
GEMM_ROUTE_SMALL_M = 2
GEMM_ROUTE_SMALL_OPERAND = 3
GEMM_ROUTE_TC_SINGLE = 4
GEMM_ROUTE_TC_PAIR = 5
GEMM_ROUTE_TINY = 6


class gemm_plan_t(ctypes.Structure):
    _fields_ = [("route", ctypes.c_int), ("bn", ctypes.c_int), ("splits", ctypes.c_int),
                ("stages", ctypes.c_int), ("grid", ctypes.c_int), ("model_us", ctypes.c_double),
                ("dram_us", ctypes.c_double), ("tail_splits", ctypes.c_int)]

_lock = threading.Lock()
_lib = None


class GemmError(RuntimeError):
    def __init__(self, status: int):
        self.status = int(status)
        super().__init__(gemm_status_string(status))


def library():
    """The loaded ``libgb300gemm.so`` (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "paper_2512_13282_gb300.build.build() (no CPU fallback exists)")
        lib = ctypes.CDLL(LIB_PATH)
        i64, vp, ci = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int
        for name in ("gemm_s8s8_s32", "gemm_bf16_f32acc_bf16", "gemm_s8s8_s32_noalloc"):
            f = getattr(lib, name)
            f.argtypes = [i64, i64, i64, vp, i64, vp, i64, ci, vp, i64, vp]
            f.restype = ci
        for name in ("gemm_s8s8_s16", "gemm_s8s8_s8"):
            f = getattr(lib, name)
            f.argtypes = [i64, i64, i64, vp, i64, vp, i64, ci, vp, i64, ci, vp]
            f.restype = ci
        lib.gemm_status_string.argtypes = [ci]
        lib.gemm_status_string.restype = ctypes.c_char_p
        lib.gemm_device_status.argtypes = []
        lib.gemm_device_status.restype = ci
        lib.gemm_release_resources.argtypes = []
        lib.gemm_release_resources.restype = None
        lib.gemm_launch_count.argtypes = []
        lib.gemm_launch_count.restype = ctypes.c_uint64
        lib.gemm_reload_overrides.argtypes = []
        lib.gemm_reload_overrides.restype = None
        lib.gemm_plan_query.argtypes = [i64, i64, i64, ci, ci, ci, ci, ctypes.POINTER(gemm_plan_t)]
        lib.gemm_plan_query.restype = ci
        lib.gemm_selftest_read_stream.argtypes = [vp, ctypes.c_size_t, vp]
        lib.gemm_selftest_read_stream.restype = ci
        lib.gemm_selftest_wait_timeout.argtypes = [ctypes.c_uint64, vp]
        lib.gemm_selftest_wait_timeout.restype = ci
        lib.gemm_profile_events.argtypes = [vp, vp]
        lib.gemm_profile_events.restype = None
        _lib = lib
        return lib


def _ptr(x) -> int:
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(s) -> int:
    if s is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


def gemm_s8s8_s32(M, N, K, A, lda, B, ldb, b_layout, C, ldc, stream=None) -> int:
    """C (int32, M x N) = A (int8, M x K) . B (int8, K x N), exact."""
    return int(library().gemm_s8s8_s32(M, N, K, _ptr(A), lda, _ptr(B), ldb, int(b_layout),
                                       _ptr(C), ldc, _stream(stream)))


def gemm_s8s8_s16(M, N, K, A, lda, B, ldb, b_layout, C, ldc, shift, stream=None) -> int:
    """C (int16) = saturate(round_half_even((A . B) / 2^shift)), A, B int8."""
    return int(library().gemm_s8s8_s16(M, N, K, _ptr(A), lda, _ptr(B), ldb, int(b_layout),
                                       _ptr(C), ldc, int(shift), _stream(stream)))


def gemm_s8s8_s8(M, N, K, A, lda, B, ldb, b_layout, C, ldc, shift, stream=None) -> int:
    """C (int8) = saturate(round_half_even((A . B) / 2^shift)), A, B int8."""
    return int(library().gemm_s8s8_s8(M, N, K, _ptr(A), lda, _ptr(B), ldb, int(b_layout),
                                      _ptr(C), ldc, int(shift), _stream(stream)))


def gemm_s8s8_s32_noalloc(M, N, K, A, lda, B, ldb, b_layout, C, ldc, stream=None) -> int:
    """gemm_s8s8_s32 for callers that cannot let the library allocate device
    memory: staging and split-K scratch live in a fixed 128 MiB device array
    (GEMM_NOALLOC_SCRATCH_BYTES); larger problems return
    GEMM_ERR_UNSUPPORTED.  Calls that overlap on the GPU race on that array."""
    return int(library().gemm_s8s8_s32_noalloc(M, N, K, _ptr(A), lda, _ptr(B), ldb, int(b_layout),
                                               _ptr(C), ldc, _stream(stream)))


def gemm_bf16_f32acc_bf16(M, N, K, A, lda, B, ldb, b_layout, C, ldc, stream=None) -> int:
    """C (bf16, M x N) = rne_bf16(A (bf16) . B (bf16)) with fp32 accumulation."""
    return int(library().gemm_bf16_f32acc_bf16(M, N, K, _ptr(A), lda, _ptr(B), ldb, int(b_layout),
                                               _ptr(C), ldc, _stream(stream)))


def gemm_status_string(status: int) -> str:
    return library().gemm_status_string(int(status)).decode()


def gemm_device_status() -> int:
    return int(library().gemm_device_status())


def gemm_release_resources() -> None:
    library().gemm_release_resources()


def gemm_launch_count() -> int:
    return int(library().gemm_launch_count())


def gemm_reload_overrides() -> None:
    """Re-read the GB300_GEMM_* planner overrides from the environment."""
    library().gemm_reload_overrides()


def gemm_selftest_wait_timeout(limit_ns: int, stream=None) -> int:
    """Launch the bounded-wait probe that is made to time out; see the header."""
    return int(library().gemm_selftest_wait_timeout(int(limit_ns), _stream(stream)))


def gemm_plan_query(M, N, K, int8, b_layout, sms=152, pair_slots=76):
    """(status, plan) of the host-only planner query; plan is a dict with
    route, bn, splits, stages, grid, model_us, dram_us and tail_splits."""
    out = gemm_plan_t()
    st = int(library().gemm_plan_query(M, N, K, 1 if int8 else 0, int(b_layout), int(sms), int(pair_slots),
                                       ctypes.byref(out)))
    return st, {f: getattr(out, f) for f, _ in gemm_plan_t._fields_}


def gemm_selftest_read_stream(ptr, nbytes, stream=None) -> int:
    """Enqueue the read-bandwidth diagnostic: a plain read of `nbytes` at
    `ptr` (device memory), results discarded; see the header."""
    return int(library().gemm_selftest_read_stream(_ptr(ptr), int(nbytes), _stream(stream)))


def gemm_profile_events(start_event, stop_event) -> None:
    """Bracket the tensor-core kernel of following calls with two CUDA
    events (``torch.cuda.Event`` or raw handles); ``None, None`` stops."""
    def h(e):
        if e is None:
            return None
        return e if isinstance(e, int) else int(e.cuda_event)
    library().gemm_profile_events(h(start_event), h(stop_event))


def check(status: int) -> None:
    if status != GEMM_OK:
        raise GemmError(status)

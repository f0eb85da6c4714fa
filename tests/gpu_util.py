"""Helpers for the GPU tests: place numpy operands in device memory with a
chosen leading dimension and base offset, call the C ABI through the binding,
and check that nothing outside [0,M) x [0,N) of C was written."""
import numpy as np
import torch

from paper_2512_13282_gb300 import gemm as G

SENTINEL32 = 0x5A5AA5A5              # fits int32
SENTINEL16 = 0x7E57                   # a NaN pattern no result can produce here


def _np_to_torch_dtype(a):
    return {np.int8: torch.int8, np.uint16: torch.int16, np.int32: torch.int32}[a.dtype.type]


def to_device(a: np.ndarray, ld: int = None, offset: int = 0):
    """Copy a 2-D host array into a fresh device buffer, row pitch `ld`
    elements, starting `offset` elements into the buffer.  Returns
    (buffer, pointer, ld)."""
    rows, cols = a.shape
    ld = max(cols, 1) if ld is None else ld
    tdt = _np_to_torch_dtype(a)
    buf = torch.zeros(offset + max(rows * ld, 1) + 16, dtype=tdt, device="cuda")
    if a.size:
        host = torch.from_numpy(np.ascontiguousarray(a).view(np.int16) if a.dtype == np.uint16
                                else np.ascontiguousarray(a))
        buf[offset:offset + rows * ld].view(rows, ld)[:, :cols].copy_(host)
    return buf, buf.data_ptr() + offset * buf.element_size(), ld


SENTINEL_S16 = 0x5A5A                 # guard values of int16 / int8 outputs
SENTINEL_S8 = 0x5A


def run(dtype, A, B, layout, lda=None, ldb=None, ldc=None, a_off=0, b_off=0, c_off=0,
        stream=None, expect=G.GEMM_OK, shift=0):
    """Run one GEMM through the C ABI.  dtype "int8" (int32 C), "int8_int16" /
    "int8_int8" (int8 operands, requantised int16 / int8 C with right shift
    `shift`) or "bf16".  Returns C (numpy int32, int16, int8 or uint16 bit patterns) after
    checking the guard region of C."""
    M, K = A.shape
    N = B.shape[1] if layout == G.GEMM_B_ROW_MAJOR_KxN else B.shape[0]
    # keep the buffers referenced until the GEMM has finished: a dropped
    # tensor's memory goes back to torch's allocator and can be handed out
    # again (e.g. to C) while the kernel still reads it
    abuf, pa, lda = to_device(A, lda, a_off)
    bbuf, pb, ldb = to_device(B, ldb, b_off)
    ldc = max(N, 1) if ldc is None else ldc
    if dtype == "int8":
        cbuf = torch.full((c_off + (M + 2) * ldc + 16,), SENTINEL32, dtype=torch.int32, device="cuda")
        fn, sent = G.gemm_s8s8_s32, SENTINEL32
    elif dtype in ("int8_int16", "int8_int8"):
        s16 = dtype == "int8_int16"
        tdt, sent = (torch.int16, SENTINEL_S16) if s16 else (torch.int8, SENTINEL_S8)
        cbuf = torch.full((c_off + (M + 2) * ldc + 16,), sent, dtype=tdt, device="cuda")
        g = G.gemm_s8s8_s16 if s16 else G.gemm_s8s8_s8

        def fn(M, N, K, pa, lda, pb, ldb, layout, pc, ldc, stream):
            return g(M, N, K, pa, lda, pb, ldb, layout, pc, ldc, shift, stream)
    else:
        cbuf = torch.full((c_off + (M + 2) * ldc + 16,), SENTINEL16, dtype=torch.int16, device="cuda")
        fn, sent = G.gemm_bf16_f32acc_bf16, SENTINEL16
    pc = cbuf.data_ptr() + c_off * cbuf.element_size()
    G.gemm_reload_overrides()  # the test may have changed GB300_GEMM_* since the last call
    st = fn(M, N, K, pa, lda, pb, ldb, layout, pc, ldc, stream)
    assert st == expect, f"status {st} ({G.gemm_status_string(st)}), expected {expect}"
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    host = cbuf.cpu().numpy()
    del abuf, bbuf
    assert (host[:c_off] == sent).all(), "bytes before C were written"
    body = host[c_off:c_off + (M + 2) * ldc].reshape(M + 2, ldc)
    assert (body[:, N:] == sent).all(), "columns past N were written"
    assert (body[M:] == sent).all(), "rows past M were written"
    assert (host[c_off + (M + 2) * ldc:] == sent).all(), "bytes after C were written"
    C = body[:M, :N].copy()
    return C.view(np.uint16) if dtype == "bf16" else C

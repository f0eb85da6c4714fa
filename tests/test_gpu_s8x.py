"""GPU parity of the int8 tensor-core kernel that converts both operands to
fp16 inside the kernel (no staging launch): exact int32 sums, and the
requantised int16 / int8 outputs, against the oracle bit for bit, with the
route forced (GB300_GEMM_S8X=1) and checked through the plan query.  Covers
ragged M, N and K (K not a multiple of the 64-deep step, and below it),
several 1024-deep exact slabs, more tiles than SMs (the persistent loop),
the int32 edge, and unaligned C (direct stores)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W
from tests import gpu_util as U

pytestmark = pytest.mark.gpu
COL = G.GEMM_B_COL_MAJOR_NxK


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


@pytest.fixture(autouse=True)
def _force(monkeypatch):
    monkeypatch.setenv("GB300_GEMM_S8X", "1")
    monkeypatch.setenv("GB300_GEMM_S8TM", "0")           # M <= 128 shapes too
    monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")  # and small problems


def _route(M, N, K):
    G.gemm_reload_overrides()
    st, plan = G.gemm_plan_query(M, N, K, True, COL)
    assert st == G.GEMM_OK
    return plan["route"]


def _check(A, B, C):
    want = oracle.gemm_s8(A, B, COL)
    bad = np.argwhere(C.astype(np.int64) != want)
    assert bad.size == 0, f"{len(bad)} mismatches, first at {bad[:5].tolist()}: " \
                          f"{C[tuple(bad[0])]} vs {want[tuple(bad[0])]}"


# (M, N, K): one tile; ragged M and N; K below one step, not a multiple of
# the step, several slabs; tiles beyond one wave (160 > 152 SMs)
SHAPES = [(128, 224, 64), (129, 225, 80), (9, 17, 16), (300, 500, 1040), (257, 449, 2064), (1000, 1500, 3008),
          (2048, 2240, 1024), (640, 7000, 512)]


@pytest.mark.parametrize("M,N,K", SHAPES, ids=[f"{m}x{n}x{k}" for m, n, k in SHAPES])
def test_s8x_parity(M, N, K):
    assert _route(M, N, K) == G.GEMM_ROUTE_TC_INT8_DIRECT
    A, B = W.random_int8((M, K), M + K), W.random_int8((N, K), N + K)
    C = U.run("int8", A, B, COL)
    _check(A, B, C)


def test_s8x_padded_pitches_and_unaligned_c():
    """K = 1001 inside pitches of 1008 bytes (the boxes read zeros past K);
    C with an odd pitch and offset takes the direct stores."""
    M, N, K = 333, 451, 1001
    A, B = W.random_int8((M, K), 3), W.random_int8((N, K), 4)
    C = U.run("int8", A, B, COL, lda=1008, ldb=1008, ldc=N + 3, c_off=1)
    _check(A, B, C)


def test_s8x_int32_edge():
    """All -128 at K = 131056: 2147221504, next to the int32 limit, through
    128 exact slabs."""
    M, N, K = 130, 230, 131056
    A = np.full((M, K), -128, np.int8)
    B = np.full((N, K), -128, np.int8)
    C = U.run("int8", A, B, COL)
    assert (C == 16384 * K).all()
    B2 = np.full((N, K), 127, np.int8)
    C2 = U.run("int8", A, B2, COL)
    assert (C2 == -16256 * K).all()


def test_s8x_every_byte_value():
    """Each of the 256 int8 values meets each other one: A's row i is the
    value i - 128 in every column, B's row j the value j - 128, so
    C[i][j] = K (i - 128)(j - 128) -- every conversion, both operands."""
    K = 64
    A = np.repeat((np.arange(256) - 128).astype(np.int8)[:, None], K, axis=1)
    B = A.copy()
    C = U.run("int8", A, B, COL)
    v = np.arange(256, dtype=np.int64) - 128
    assert np.array_equal(C.astype(np.int64), K * np.outer(v, v))


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
def test_s8x_requantised_outputs(out):
    bits = 16 if out == "int8_int16" else 8
    M, N, K = 300, 700, 2048
    A, B = W.random_int8((M, K), 11), W.random_int8((N, K), 12)
    shift = max(0, int(np.log2(5500.0 * np.sqrt(K))) + 2 - bits)
    C = U.run(out, A, B, COL, shift=shift)
    want = oracle.requantize(oracle.gemm_s8(A, B, COL), shift, bits)
    assert np.array_equal(C.astype(np.int64), want)


def test_s8x_not_taken_where_illegal(monkeypatch):
    """B stored K x N, or pitches that are not a multiple of 16 bytes: the
    kernel's boxes cannot be described, so the staged path runs instead
    (and is exact)."""
    assert G.gemm_plan_query(500, 600, 700, True, G.GEMM_B_ROW_MAJOR_KxN)[1]["route"] != \
        G.GEMM_ROUTE_TC_INT8_DIRECT
    assert _route(500, 600, 1000) != G.GEMM_ROUTE_TC_INT8_DIRECT  # K % 16 != 0: tight pitches unaligned
    M, N, K = 200, 300, 1000
    A, B = W.random_int8((M, K), 21), W.random_int8((N, K), 22)
    C = U.run("int8", A, B, COL)
    _check(A, B, C)

"""GPU parity of the reduced-precision int8 outputs (int8-int16 and
int8-int8, Sec. 5.1): every element must equal the oracle's
saturate(round_half_even(exact_sum / 2^shift)) bit for bit, on every path
that forms the sum -- single-CTA and CTA-pair tensor-core kernels, split-K
with its reduction pass, the CUDA-core small-M kernel -- with ragged edges,
unaligned C rows and K = 0."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W
from tests import gpu_util as U

pytestmark = pytest.mark.gpu
ROW, COL = G.GEMM_B_ROW_MAJOR_KxN, G.GEMM_B_COL_MAJOR_NxK
BITS = {"int8_int16": 16, "int8_int8": 8}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


def _inputs(M, N, K, layout, seed):
    bshape = (K, N) if layout == ROW else (N, K)
    return W.random_int8((M, K), seed), W.random_int8(bshape, seed + 1)


def _check(out, A, B, layout, shift, C):
    want = oracle.requantize(oracle.gemm_s8(A, B, layout), shift, BITS[out])
    bad = np.argwhere(C.astype(np.int64) != want)
    assert bad.size == 0, f"{len(bad)} mismatches, first at {bad[:5].tolist()}: " \
                          f"{C[tuple(bad[0])]} vs {want[tuple(bad[0])]}"
    return want


def _shift_for(out, K):
    # keeps most sums inside the output range (|sum| ~ 74^2 * sqrt(K)) while
    # some still saturate and rounding still has ties to settle
    return max(0, int(np.log2(5500.0 * np.sqrt(max(K, 1)))) + 2 - BITS[out])


SHAPES = [(1, 1, 1), (5, 7, 3), (129, 257, 65), (300, 520, 200), (1000, 1500, 3000), (257, 129, 2100)]


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", SHAPES, ids=[f"{m}x{n}x{k}" for m, n, k in SHAPES])
@pytest.mark.parametrize("path", ["auto", "tensor"])
def test_requant_parity_shapes(out, layout, M, N, K, path, monkeypatch):
    if path == "tensor":
        monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    A, B = _inputs(M, N, K, layout, seed=M + 5 * N + 7 * K)
    shift = _shift_for(out, K)
    C = U.run(out, A, B, layout, shift=shift)
    want = _check(out, A, B, layout, shift, C)
    if M * N >= 10000:  # the shift chosen leaves both saturated and in-range results
        lim = 2 ** (BITS[out] - 1)
        assert (np.abs(want) < lim - 1).mean() > 0.5


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("shift", [0, 1, 7, 13, 31])
def test_requant_every_shift_class(out, layout, shift):
    A, B = _inputs(200, 300, 1100, layout, seed=shift + 3)
    C = U.run(out, A, B, layout, shift=shift)
    _check(out, A, B, layout, shift, C)


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("bn", [128, 192, 224, 256])
@pytest.mark.parametrize("pair", ["0", "1"], ids=["single", "pair"])
def test_requant_every_tile_width(out, layout, bn, pair, monkeypatch):
    if layout == ROW and bn == 224:
        pytest.skip("no 224-wide tile for row-major B")
    if layout == ROW and pair == "1" and bn == 192:
        pytest.skip("pairs with row-major B use 128 or 256")
    monkeypatch.setenv("GB300_GEMM_BN", str(bn))
    monkeypatch.setenv("GB300_GEMM_PAIR", pair)
    A, B = _inputs(600, 900, 1500, layout, seed=bn)
    shift = _shift_for(out, 1500)
    C = U.run(out, A, B, layout, shift=shift)
    _check(out, A, B, layout, shift, C)


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", [(16, 512, 4096), (130, 300, 9000)])
def test_requant_split_k(out, layout, M, N, K, monkeypatch):
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    monkeypatch.setenv("GB300_GEMM_SPLITS", "5")
    A, B = _inputs(M, N, K, layout, seed=K)
    shift = _shift_for(out, K)
    C = U.run(out, A, B, layout, shift=shift)
    _check(out, A, B, layout, shift, C)


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", [(1, 1000, 777), (3, 4100, 4096), (8, 300, 20000)])
def test_requant_small_m(out, layout, M, N, K):
    A, B = _inputs(M, N, K, layout, seed=M + K)
    shift = _shift_for(out, K)
    C = U.run(out, A, B, layout, shift=shift)
    _check(out, A, B, layout, shift, C)


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M", [4, 300])
@pytest.mark.parametrize("path", ["auto", "tensor"])
def test_requant_unaligned_c(out, layout, M, path, monkeypatch):
    # odd ldc and a C base 1 element past an aligned address: every row
    # starts at a different alignment, so all store widths are used
    if path == "tensor":
        monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    A, B = _inputs(M, 517, 640, layout, seed=M)
    shift = _shift_for(out, 640)
    C = U.run(out, A, B, layout, ldc=523, c_off=1, shift=shift)
    _check(out, A, B, layout, shift, C)


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
def test_requant_extremes_and_ties(out):
    # all -128 with K = 64: every sum is 2^20; shifts 19 and 20 give 2 and 1
    # exactly, 21 a tie (0.5 -> 0), 0 saturates.  A second problem puts
    # exact .5 ties next to both odd and even quotients.
    K = 64
    A = np.full((200, K), -128, np.int8)
    B = np.full((K, 300), -128, np.int8)
    for shift in (19, 20, 21, 0):
        C = U.run(out, A, B, ROW, shift=shift)
        _check(out, A, B, ROW, shift, C)
    A = np.zeros((150, 2), np.int8)
    A[:, 0] = np.arange(150) - 75
    A[:, 1] = 1
    B = np.array([[2] * 260, [1] * 260], np.int8)  # sums 2a + 1: odd, ties at shift 1
    C = U.run(out, A, B, ROW, shift=1)
    want = _check(out, A, B, ROW, 1, C)
    assert set(np.unique(want[:, 0] % 2)) == {0}  # ties went to even


@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
def test_requant_k_zero(out):
    A = np.zeros((7, 0), np.int8)
    B = np.zeros((0, 9), np.int8)
    C = U.run(out, A, B, ROW, shift=5)
    assert (C == 0).all()


def test_requant_consistent_with_int32_path():
    # the narrow outputs are the int32 path's results requantised
    A, B = _inputs(700, 1100, 2000, COL, seed=77)
    C32 = U.run("int8", A, B, COL)
    for out, shift in (("int8_int16", 4), ("int8_int8", 12)):
        C = U.run(out, A, B, COL, shift=shift)
        assert np.array_equal(C.astype(np.int64), oracle.requantize(C32.astype(np.int64), shift, BITS[out]))


DIRECT_CASES = [(300, 700, 1500, "1", None, 0), (130, 450, 3000, "3", None, 0), (300, 517, 640, "1", 523, 1),
                (257, 333, 2100, "2", None, 0)]
DIRECT_KERNELS = [(192, "0", ROW), (192, "0", COL), (224, "0", COL), (192, "1", COL), (224, "1", COL),
                  (128, "0", COL), (256, "1", ROW)]


@pytest.mark.parametrize("out", ["int8", "int8_int16", "int8_int8"])
@pytest.mark.parametrize("bn,pair,layout", DIRECT_KERNELS,
                         ids=[f"{b}-{'pair' if p == '1' else 'single'}-{'Brow' if l == ROW else 'Bcol'}"
                              for b, p, l in DIRECT_KERNELS])
def test_int8_direct_stores(out, bn, pair, layout, monkeypatch):
    """The int8 epilogue without TMA stores (the direct-store kernels with
    the extra pipeline stage at 192 / 224, the TMA kernels' fallback at 128 /
    256): int32 and requantised C, split-K partials (including a pitch N that
    is not a multiple of 4), ragged edges and unaligned C rows."""
    monkeypatch.setenv("GB300_GEMM_TMA_STORE", "0")
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    monkeypatch.setenv("GB300_GEMM_BN", str(bn))
    monkeypatch.setenv("GB300_GEMM_PAIR", pair)
    for (M, N, K, splits, ldc, c_off) in DIRECT_CASES:
        monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
        A, B = _inputs(M, N, K, layout, seed=M + N + bn)
        if out == "int8":
            C = U.run(out, A, B, layout, ldc=ldc, c_off=c_off)
            want = oracle.gemm_s8(A, B, layout)
            assert np.array_equal(C.astype(np.int64), want), (M, N, K, splits)
        else:
            shift = _shift_for(out, K)
            C = U.run(out, A, B, layout, ldc=ldc, c_off=c_off, shift=shift)
            _check(out, A, B, layout, shift, C)

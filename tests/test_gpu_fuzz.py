"""GPU parity on seeded random problems: random shapes (log-uniform M, N, K,
from single elements to a few tiles with ragged edges), both B layouts, all
four output types, random leading-dimension padding and base offsets, and a
random route forced now and then (the CUDA-core small-M and tiny kernels on
or off, the small-operand int8 kernel off, a tile width, a K split) --
every element against the oracle (int8 exact, bf16 within the bound and the
rounding check).  The cases are fixed by the seed, so a failure names a
reproducible case."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W
from tests import gpu_util as U
from tests.test_gpu_parity import _check_rounding

pytestmark = pytest.mark.gpu
ROW, COL = G.GEMM_B_ROW_MAJOR_KxN, G.GEMM_B_COL_MAJOR_NxK
ROUTE_ENV = ("GB300_GEMM_SKINNY_MAX_M", "GB300_GEMM_TINY_MAX_MACS", "GB300_GEMM_S8TM", "GB300_GEMM_BN",
             "GB300_GEMM_SPLITS", "GB300_GEMM_PAIR")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


def _case(i):
    """Case i: (dtype, layout, M, N, K, pads, offsets, env, shift)."""
    rng = np.random.default_rng(1000 + i)
    big = rng.uniform() < 0.5  # several tiles, or log-uniform from 1 (edges, tiny and skinny problems)
    while True:
        if not big:
            M, N, K = (int(round(np.exp(rng.uniform(0, np.log(hi))))) for hi in (900, 1100, 2500))
        else:
            M, N, K = (int(rng.integers(lo, hi)) for lo, hi in ((100, 900), (100, 1100), (64, 2500)))
        if M * N * K <= 1.5e8:
            break
    dtype = ("int8", "bf16", "int8_int16", "int8_int8")[i % 4]
    layout = (ROW, COL)[(i // 4) % 2]
    pads = tuple(int(x) for x in rng.choice([0, 0, 1, 3, 8, 17], 3))
    offs = tuple(int(x) for x in rng.choice([0, 0, 1, 2], 3))
    env = {}
    r = rng.uniform()
    if r < 0.15:
        env["GB300_GEMM_SKINNY_MAX_M"] = "16"
    elif r < 0.30:
        env["GB300_GEMM_SKINNY_MAX_M"] = "0"
        env["GB300_GEMM_TINY_MAX_MACS"] = "0"
        env["GB300_GEMM_S8TM"] = "0"
    elif r < 0.45:
        env["GB300_GEMM_TINY_MAX_MACS"] = "0"
        env["GB300_GEMM_BN"] = str(int(rng.choice([128, 192, 224, 256])))
        env["GB300_GEMM_SPLITS"] = str(int(rng.integers(1, 5)))
        env["GB300_GEMM_PAIR"] = str(int(rng.integers(0, 2)))
    shift = int(rng.integers(0, 12)) if dtype in ("int8_int16", "int8_int8") else 0
    return dtype, layout, M, N, K, pads, offs, env, shift


CASES = [_case(i) for i in range(200)]


@pytest.mark.parametrize("i", range(len(CASES)),
                         ids=[f"{c[0]}-{'Brow' if c[1] == ROW else 'Bcol'}-{c[2]}x{c[3]}x{c[4]}" for c in CASES])
def test_fuzz(i, monkeypatch):
    dtype, layout, M, N, K, pads, offs, env, shift = CASES[i]
    for k in ROUTE_ENV:
        monkeypatch.delenv(k, raising=False)
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    seed = 7 * i + 1
    bshape = (K, N) if layout == ROW else (N, K)
    if dtype == "bf16":
        A, B = W.random_bf16((M, K), seed), W.random_bf16(bshape, seed + 1)
    else:
        A, B = W.random_int8((M, K), seed), W.random_int8(bshape, seed + 1)
    bcols = N if layout == ROW else K
    C = U.run(dtype, A, B, layout, lda=K + pads[0], ldb=bcols + pads[1], ldc=N + pads[2], a_off=offs[0],
              b_off=offs[1], c_off=offs[2], shift=shift)
    if dtype == "bf16":
        ref, mag = oracle.gemm_bf16(A, B, layout)
        ok = oracle.bf16_within_bound(C, ref, mag)
        assert ok.all(), f"{np.sum(~ok)} elements out of bound"
        _check_rounding(C, ref)
    else:
        want = oracle.gemm_s8(A, B, layout)
        if dtype != "int8":
            want = oracle.requantize(want, shift, 16 if dtype == "int8_int16" else 8)
        bad = np.argwhere(C.astype(np.int64) != want)
        assert bad.size == 0, f"{len(bad)} mismatches, first at {bad[:5].tolist()}"


def _case_small_operand(i):
    """Shapes of the small-operand int8 kernel: one side of at most 128 rows
    against a long other side, K across several 1024-deep slabs, B in both
    layouts, with padded pitches (multiples of 16 bytes, so that the
    operands stay TMA-legal) or odd ones (the general path then)."""
    rng = np.random.default_rng(5000 + i)
    small = int(rng.integers(1, 129))
    big = int(rng.integers(129, 3000))
    K = int(rng.integers(16, 6000))
    if i % 3 == 2:  # N is the small side
        M, N = big, small
    else:
        M, N = small, big
    while M * N * K > 2e8:
        K //= 2
    layout = (ROW, COL)[i % 2]
    out = ("int8", "int8_int16", "int8_int8")[(i // 2) % 3]
    aligned = rng.uniform() < 0.7
    pad = lambda n: (-n) % 16 + 16 * int(rng.integers(0, 2)) if aligned else int(rng.integers(0, 5))
    return out, layout, M, N, K, pad, int(rng.integers(0, 12))


SMALL_OPERAND = [_case_small_operand(i) for i in range(90)]


@pytest.mark.parametrize("i", range(len(SMALL_OPERAND)),
                         ids=[f"{c[0]}-{'Brow' if c[1] == ROW else 'Bcol'}-{c[2]}x{c[3]}x{c[4]}" for c in SMALL_OPERAND])
def test_fuzz_small_operand(i, monkeypatch):
    out, layout, M, N, K, pad, shift = SMALL_OPERAND[i]
    for k in ROUTE_ENV:
        monkeypatch.delenv(k, raising=False)
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    A = W.random_int8((M, K), 3 * i + 1)
    B = W.random_int8((K, N) if layout == ROW else (N, K), 3 * i + 2)
    bcols = N if layout == ROW else K
    lda, ldb = K + pad(K), bcols + pad(bcols)
    shift = shift if out != "int8" else 0
    C = U.run(out, A, B, layout, lda=lda, ldb=ldb, shift=shift)
    want = oracle.gemm_s8(A, B, layout)
    if out != "int8":
        want = oracle.requantize(want, shift, 16 if out == "int8_int16" else 8)
    bad = np.argwhere(C.astype(np.int64) != want)
    assert bad.size == 0, f"{len(bad)} mismatches, first at {bad[:5].tolist()}"


def _case_noalloc(i):
    rng = np.random.default_rng(9000 + i)
    M, N, K = (int(np.exp(rng.uniform(np.log(lo), np.log(hi)))) for lo, hi in ((1, 700), (1, 900), (1, 3000)))
    return M, N, K, (ROW, COL)[i % 2], int(rng.integers(0, 3))


NOALLOC = [_case_noalloc(i) for i in range(24)]


@pytest.mark.parametrize("i", range(len(NOALLOC)),
                         ids=[f"{'Brow' if c[3] == ROW else 'Bcol'}-{c[0]}x{c[1]}x{c[2]}" for c in NOALLOC])
def test_fuzz_noalloc(i):
    """The no-allocation entry point on random shapes, padded pitches and
    offsets, against the oracle."""
    M, N, K, layout, pad = NOALLOC[i]
    A = W.random_int8((M, K), 11 * i + 1)
    B = W.random_int8((K, N) if layout == ROW else (N, K), 11 * i + 2)
    bcols = N if layout == ROW else K
    abuf, pa, lda = U.to_device(A, K + pad, pad)
    bbuf, pb, ldb = U.to_device(B, bcols + pad, 0)
    ldc = N + pad
    C = torch.full((M * ldc + 16,), U.SENTINEL32, dtype=torch.int32, device="cuda")
    st = G.gemm_s8s8_s32_noalloc(M, N, K, pa, lda, pb, ldb, layout, C.data_ptr(), ldc, 0)
    assert st == G.GEMM_OK, G.gemm_status_string(st)
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    host = C.cpu().numpy()
    body = host[:M * ldc].reshape(M, ldc)
    assert (body[:, N:] == U.SENTINEL32).all() and (host[M * ldc:] == U.SENTINEL32).all()
    assert np.array_equal(body[:, :N].astype(np.int64), oracle.gemm_s8(A, B, layout))
    del abuf, bbuf


def _case_large(i):
    """More tiles than SMs (persistent loops over several rounds, group
    rasterisation edges), with a forced family / width / split now and then."""
    rng = np.random.default_rng(7000 + i)
    M, N, K = int(rng.integers(1200, 3000)), int(rng.integers(1200, 3000)), int(rng.integers(200, 900))
    dtype = ("int8", "bf16")[i % 2]
    layout = (ROW, COL)[(i // 2) % 2]
    env = {}
    if i % 3 == 1:
        env = {"GB300_GEMM_BN": str(int(rng.choice([128, 192, 224, 256]))),
               "GB300_GEMM_PAIR": str(int(rng.integers(0, 2))), "GB300_GEMM_SPLITS": str(int(rng.integers(1, 4)))}
    return dtype, layout, M, N, K, env


LARGE = [_case_large(i) for i in range(12)]


@pytest.mark.parametrize("i", range(len(LARGE)),
                         ids=[f"{c[0]}-{'Brow' if c[1] == ROW else 'Bcol'}-{c[2]}x{c[3]}x{c[4]}" for c in LARGE])
def test_fuzz_large(i, monkeypatch):
    dtype, layout, M, N, K, env = LARGE[i]
    for k in ROUTE_ENV:
        monkeypatch.delenv(k, raising=False)
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    bshape = (K, N) if layout == ROW else (N, K)
    if dtype == "bf16":
        A, B = W.random_bf16((M, K), 13 * i + 1), W.random_bf16(bshape, 13 * i + 2)
    else:
        A, B = W.random_int8((M, K), 13 * i + 1), W.random_int8(bshape, 13 * i + 2)
    C = U.run(dtype, A, B, layout)
    if dtype == "bf16":
        ref, mag = oracle.gemm_bf16(A, B, layout)
        assert oracle.bf16_within_bound(C, ref, mag).all()
        _check_rounding(C, ref)
    else:
        assert np.array_equal(C.astype(np.int64), oracle.gemm_s8(A, B, layout))


def _case_aspect(i):
    """Extreme aspect ratios: one of M, N, K tiny (1..16) against the others."""
    rng = np.random.default_rng(8000 + i)
    dims = [int(rng.integers(1, 17)), int(rng.integers(200, 4000)), int(rng.integers(200, 4000))]
    rng.shuffle(dims)
    M, N, K = dims
    while M * N * K > 1.2e8:
        K = max(1, K // 2)
    return ("int8", "bf16")[i % 2], (ROW, COL)[(i // 2) % 2], M, N, K


ASPECT = [_case_aspect(i) for i in range(40)]


@pytest.mark.parametrize("i", range(len(ASPECT)),
                         ids=[f"{c[0]}-{'Brow' if c[1] == ROW else 'Bcol'}-{c[2]}x{c[3]}x{c[4]}" for c in ASPECT])
def test_fuzz_aspect(i, monkeypatch):
    dtype, layout, M, N, K = ASPECT[i]
    for k in ROUTE_ENV:
        monkeypatch.delenv(k, raising=False)
    bshape = (K, N) if layout == ROW else (N, K)
    if dtype == "bf16":
        A, B = W.random_bf16((M, K), 17 * i + 1), W.random_bf16(bshape, 17 * i + 2)
    else:
        A, B = W.random_int8((M, K), 17 * i + 1), W.random_int8(bshape, 17 * i + 2)
    C = U.run(dtype, A, B, layout)
    if dtype == "bf16":
        ref, mag = oracle.gemm_bf16(A, B, layout)
        assert oracle.bf16_within_bound(C, ref, mag).all()
        _check_rounding(C, ref)
    else:
        assert np.array_equal(C.astype(np.int64), oracle.gemm_s8(A, B, layout))

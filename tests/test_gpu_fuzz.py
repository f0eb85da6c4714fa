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

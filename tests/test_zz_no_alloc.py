"""gemm_s8s8_s32_noalloc: the int8 GEMM for callers that cannot let the
library allocate device memory (their own allocator already holds the GPU's
memory, they enforce a strict memory budget, or they cannot absorb
cudaMalloc's latency and synchronisation).

It must give exactly the results of gemm_s8s8_s32 and of the oracle (int8
results are exact, so the comparisons are bit for bit), also when called
twice in a row on different problems -- the second call reuses the fixed
scratch array the first one left behind -- and it must reject problems
larger than its scratch without launching anything.  The array is reserved
on the GPU by the first call, and by no later one.  Named test_zz_* so that
pytest collects it last.
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


def _operands(M, N, K, layout, seed):
    A = torch.from_numpy(W.random_int8((M, K), seed)).cuda()
    bshape = (K, N) if layout == G.GEMM_B_ROW_MAJOR_KxN else (N, K)
    B = torch.from_numpy(W.random_int8(bshape, seed + 1)).cuda()
    ldb = N if layout == G.GEMM_B_ROW_MAJOR_KxN else K
    return A, B, ldb


def test_noalloc_matches_allocating_entry_point_twice_in_a_row():
    problems = [(300, 520, 2100, G.GEMM_B_COL_MAJOR_NxK, 7),    # split-K partials in scratch
                (64, 1000, 1100, G.GEMM_B_ROW_MAJOR_KxN, 11)]   # different layout and sizes
    results = []
    for (M, N, K, layout, seed) in problems:
        A, B, ldb = _operands(M, N, K, layout, seed)
        C_ref = torch.empty((M, N), dtype=torch.int32, device="cuda")
        G.check(G.gemm_s8s8_s32(M, N, K, A, K, B, ldb, layout, C_ref, N))
        C_new = torch.full((M, N), -7, dtype=torch.int32, device="cuda")
        results.append((A, B, ldb, layout, M, N, K, C_ref, C_new))
    torch.cuda.synchronize()
    # two no-allocation calls back to back on the same stream
    for (A, B, ldb, layout, M, N, K, C_ref, C_new) in results:
        G.check(G.gemm_s8s8_s32_noalloc(M, N, K, A, K, B, ldb, layout, C_new, N))
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    for (A, B, ldb, layout, M, N, K, C_ref, C_new) in results:
        assert torch.equal(C_new, C_ref), f"{M}x{N}x{K}: no-allocation result differs"
        want = oracle.gemm_s8(A.cpu().numpy(), B.cpu().numpy(), layout)
        assert np.array_equal(C_new.cpu().numpy().astype(np.int64), want), f"{M}x{N}x{K}: differs from the oracle"


_FRESH_PROCESS = r"""
import sys, torch
sys.path.insert(0, sys.argv[1])
from paper_2512_13282_gb300 import build, gemm as G
from paper_2512_13282_gb300 import workloads as W
build.build()
torch.cuda.init()
M, N, K = 256, 384, 3000
A = torch.from_numpy(W.random_int8((M, K), 5)).cuda()
B = torch.from_numpy(W.random_int8((N, K), 6)).cuda()
C = torch.empty((M, N), dtype=torch.int32, device="cuda")
# load the kernels' code and the workspace through the allocating entry point first
G.check(G.gemm_s8s8_s32(M, N, K, A, K, B, K, G.GEMM_B_COL_MAJOR_NxK, C, N))
torch.cuda.synchronize()
drops = []
for _ in range(3):
    f0 = torch.cuda.mem_get_info()[0]
    G.check(G.gemm_s8s8_s32_noalloc(M, N, K, A, K, B, K, G.GEMM_B_COL_MAJOR_NxK, C, N))
    torch.cuda.synchronize()
    drops.append(f0 - torch.cuda.mem_get_info()[0])
print(" ".join(str(d) for d in drops))
"""


def test_noalloc_first_call_reserves_the_scratch_and_later_calls_nothing():
    """In a fresh process: the first no-allocation call takes the scratch
    array's memory from the GPU (the caller must make it before its own
    allocator claims the device), the next calls take nothing."""
    out = subprocess.run([sys.executable, "-c", _FRESH_PROCESS, ROOT], capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    drops = [int(x) for x in out.stdout.split()[-3:]]
    scratch = G.GEMM_NOALLOC_SCRATCH_BYTES
    assert scratch <= drops[0] <= scratch + (8 << 20), drops
    assert drops[1] == 0 and drops[2] == 0, drops


def test_noalloc_leaves_free_memory_unchanged():
    M, N, K = 256, 384, 3000
    A, B, ldb = _operands(M, N, K, G.GEMM_B_COL_MAJOR_NxK, 21)
    C1 = torch.empty((M, N), dtype=torch.int32, device="cuda")
    C2 = torch.empty((M, N), dtype=torch.int32, device="cuda")
    G.check(G.gemm_s8s8_s32_noalloc(M, N, K, A, K, B, ldb, G.GEMM_B_COL_MAJOR_NxK, C1, N))
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    G.check(G.gemm_s8s8_s32_noalloc(M, N, K, A, K, B, ldb, G.GEMM_B_COL_MAJOR_NxK, C2, N))
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert torch.equal(C1, C2)


def test_noalloc_rejects_problems_beyond_its_scratch():
    M = N = K = 8192   # bf16 staging of A and B alone needs 256 MiB > 128 MiB
    A = torch.zeros((M, K), dtype=torch.int8, device="cuda")
    B = torch.zeros((N, K), dtype=torch.int8, device="cuda")
    C = torch.full((M, N), 5, dtype=torch.int32, device="cuda")
    st = G.gemm_s8s8_s32_noalloc(M, N, K, A, K, B, K, G.GEMM_B_COL_MAJOR_NxK, C, N)
    assert st == G.GEMM_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert bool((C == 5).all()), "a rejected call must not write C"

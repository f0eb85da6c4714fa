"""Concurrent calls on several streams: every stream has scratch of its
own, so GEMMs that stage operands, write split-K partials or use the small-M
kernel's counters may overlap on the GPU.  Each stream first runs a ~1 ms
spin kernel, so that all streams' GEMMs are queued before any starts and
then run together; every result is compared with the oracle.  A second test
uses more streams than the library keeps scratch slots for (per-call
scratch)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W
from tests import gpu_util as U

pytestmark = pytest.mark.gpu
ROW, COL = G.GEMM_B_ROW_MAJOR_KxN, G.GEMM_B_COL_MAJOR_NxK


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


# (dtype, M, N, K, layout): int8 staged (tensor path; few tiles and long K,
# so split-K grids of well under 152 CTAs let several streams' kernels share
# the GPU), int8 with one small operand, bf16 with split-K partials, the
# small-M kernel with K slices (counters)
JOBS = [("int8", 256, 300, 6000, COL), ("int8", 300, 260, 6000, ROW), ("int8", 96, 3000, 2048, COL),
        ("bf16", 200, 300, 6000, ROW), ("int8", 4, 3000, 3000, ROW), ("bf16", 2, 2500, 3000, COL)]


def _enqueue(job, seed, stream, keep):
    dtype, M, N, K, layout = job
    bshape = (K, N) if layout == ROW else (N, K)
    if dtype == "int8":
        A, B = W.random_int8((M, K), seed), W.random_int8(bshape, seed + 1)
        tA, tB = torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda()
        C = torch.zeros((M, N), dtype=torch.int32, device="cuda")
        fn = G.gemm_s8s8_s32
    else:
        A, B = W.random_bf16((M, K), seed), W.random_bf16(bshape, seed + 1)
        tA = torch.from_numpy(A.view(np.int16)).cuda()
        tB = torch.from_numpy(B.view(np.int16)).cuda()
        C = torch.zeros((M, N), dtype=torch.int16, device="cuda")
        fn = G.gemm_bf16_f32acc_bf16
    keep.append((tA, tB))
    ldb = N if layout == ROW else K
    st = fn(M, N, K, tA.data_ptr(), K, tB.data_ptr(), ldb, layout, C.data_ptr(), N, stream.cuda_stream)
    assert st == G.GEMM_OK, G.gemm_status_string(st)
    return (job, A, B, C)


def _check(job, A, B, C):
    dtype, M, N, K, layout = job
    if dtype == "int8":
        assert np.array_equal(C.cpu().numpy().astype(np.int64), oracle.gemm_s8(A, B, layout)), job
    else:
        ref, mag = oracle.gemm_bf16(A, B, layout)
        assert oracle.bf16_within_bound(C.cpu().numpy().view(np.uint16), ref, mag).all(), job


@pytest.mark.parametrize("nstreams", [2, 4])
def test_streams_concurrent(nstreams):
    G.gemm_reload_overrides()
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in range(nstreams)]
    keep, outs = [], []
    for s in streams:
        with torch.cuda.stream(s):
            torch.cuda._sleep(2_000_000)
    for j, job in enumerate(JOBS):  # round-robin: the same job type on every stream at once
        for i, s in enumerate(streams):
            outs.append(_enqueue(job, 100 * i + 7 * j, s, keep))
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    for o in outs:
        _check(*o)


def test_more_streams_than_slots():
    """20 streams: the first 16 keep scratch slots (possibly from earlier
    tests), the rest allocate scratch per call; all run together."""
    G.gemm_reload_overrides()
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in range(20)]
    keep, outs = [], []
    for s in streams:
        with torch.cuda.stream(s):
            torch.cuda._sleep(1_000_000)
    for i, s in enumerate(streams):
        outs.append(_enqueue(JOBS[i % 2], 31 * i + 5, s, keep))
        outs.append(_enqueue(JOBS[4], 31 * i + 9, s, keep))
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    for o in outs:
        _check(*o)


def test_streams_stress_against_single_calls():
    """Eight streams, each with GEMMs that stage operands and write split-K
    partials (int8 and bf16), queued together behind a spin kernel; every
    result must equal the same GEMM run alone (the library's results are
    deterministic, bf16 included).  A build that shared one workspace
    between streams got 90 of 96 such int8 results wrong."""
    G.gemm_reload_overrides()
    jobs = [("int8", 1024, 1024, 8192, COL), ("int8", 512, 2048, 4096, ROW), ("int8", 256, 300, 6000, COL),
            ("bf16", 200, 300, 6000, ROW), ("bf16", 1500, 700, 3000, COL)]
    streams = [torch.cuda.Stream() for _ in range(8)]
    items = []
    for i, s in enumerate(streams):
        for j, (dtype, M, N, K, layout) in enumerate(jobs):
            seed = 100 * i + j
            bsh = (K, N) if layout == ROW else (N, K)
            if dtype == "int8":
                tA = torch.from_numpy(W.random_int8((M, K), seed)).cuda()
                tB = torch.from_numpy(W.random_int8(bsh, seed + 1)).cuda()
                fn, cdt = G.gemm_s8s8_s32, torch.int32
            else:
                tA = torch.from_numpy(W.random_bf16((M, K), seed).view(np.int16)).cuda()
                tB = torch.from_numpy(W.random_bf16(bsh, seed + 1).view(np.int16)).cuda()
                fn, cdt = G.gemm_bf16_f32acc_bf16, torch.int16
            items.append((s, fn, cdt, M, N, K, layout, tA, tB))

    def call(it, stream):
        s, fn, cdt, M, N, K, layout, tA, tB = it
        C = torch.zeros((M, N), dtype=cdt, device="cuda")
        st = fn(M, N, K, tA.data_ptr(), K, tB.data_ptr(), N if layout == ROW else K, layout, C.data_ptr(), N,
                stream.cuda_stream)
        assert st == G.GEMM_OK, G.gemm_status_string(st)
        return C

    cur = torch.cuda.current_stream()
    alone = []
    for it in items:
        alone.append(call(it, cur))
        torch.cuda.synchronize()
    for s in streams:
        with torch.cuda.stream(s):
            torch.cuda._sleep(3_000_000)
    together = [call(it, it[0]) for it in items]
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    bad = [k for k, (a, b) in enumerate(zip(alone, together)) if not torch.equal(a, b)]
    assert not bad, f"{len(bad)} of {len(items)} concurrent GEMMs differ from the same GEMM run alone"


def test_host_threads_each_with_a_stream():
    """Four host threads, each issuing GEMMs on a stream of its own at the
    same time (the binding releases the interpreter lock inside each call):
    every result equals the same GEMM run alone."""
    import threading
    G.gemm_reload_overrides()
    jobs = [("int8", 700, 800, 3000, COL), ("bf16", 200, 300, 6000, ROW), ("int8", 4, 3000, 3000, ROW),
            ("int8", 96, 3000, 2048, COL)]
    per_thread = []
    for t in range(4):
        items = []
        for j, (dtype, M, N, K, layout) in enumerate(jobs):
            seed = 50 * t + j
            bsh = (K, N) if layout == ROW else (N, K)
            if dtype == "int8":
                tA = torch.from_numpy(W.random_int8((M, K), seed)).cuda()
                tB = torch.from_numpy(W.random_int8(bsh, seed + 1)).cuda()
                fn, cdt = G.gemm_s8s8_s32, torch.int32
            else:
                tA = torch.from_numpy(W.random_bf16((M, K), seed).view(np.int16)).cuda()
                tB = torch.from_numpy(W.random_bf16(bsh, seed + 1).view(np.int16)).cuda()
                fn, cdt = G.gemm_bf16_f32acc_bf16, torch.int16
            items.append((fn, cdt, M, N, K, layout, tA, tB))
        per_thread.append(items)

    def call(it, stream):
        fn, cdt, M, N, K, layout, tA, tB = it
        C = torch.zeros((M, N), dtype=cdt, device="cuda")
        st = fn(M, N, K, tA.data_ptr(), K, tB.data_ptr(), N if layout == ROW else K, layout, C.data_ptr(), N,
                stream.cuda_stream)
        return st, C

    cur = torch.cuda.current_stream()
    alone = [[call(it, cur)[1] for it in items] for items in per_thread]
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in range(4)]
    results = [None] * 4
    start = threading.Barrier(4)

    def worker(t):
        start.wait()
        out = []
        for _ in range(3):
            out += [call(it, streams[t]) for it in per_thread[t]]
        results[t] = out

    threads = [threading.Thread(target=worker, args=(t,)) for t in range(4)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    for t in range(4):
        for k, (st, C) in enumerate(results[t]):
            assert st == G.GEMM_OK
            assert torch.equal(C, alone[t][k % len(jobs)]), (t, k)

"""GEMM calls captured into a CUDA graph: after the stream has run the same
calls once, a graph of int8 (staged and small-operand), bf16 split-K and
small-M GEMMs replays correctly with new operand values written into the
same buffers, keeps working after a larger call on the stream grows its
scratch, and a captured call that would need more scratch is refused before
enqueuing anything."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W

pytestmark = pytest.mark.gpu
ROW, COL = G.GEMM_B_ROW_MAJOR_KxN, G.GEMM_B_COL_MAJOR_NxK


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


JOBS = [("int8", 600, 900, 1000, COL), ("int8", 96, 3000, 2048, COL), ("bf16", 200, 300, 6000, ROW),
        ("int8", 4, 3000, 3000, ROW), ("bf16", 700, 500, 1000, COL)]


class Job:
    def __init__(self, dtype, M, N, K, layout):
        self.dtype, self.M, self.N, self.K, self.layout = dtype, M, N, K, layout
        bsh = (K, N) if layout == ROW else (N, K)
        tdt = torch.int8 if dtype == "int8" else torch.int16
        self.A = torch.zeros((M, K), dtype=tdt, device="cuda")
        self.B = torch.zeros(bsh, dtype=tdt, device="cuda")
        self.C = torch.zeros((M, N), dtype=torch.int32 if dtype == "int8" else torch.int16, device="cuda")

    def fill(self, seed):
        bsh = tuple(self.B.shape)
        if self.dtype == "int8":
            self.a, self.b = W.random_int8((self.M, self.K), seed), W.random_int8(bsh, seed + 1)
            self.A.copy_(torch.from_numpy(self.a)); self.B.copy_(torch.from_numpy(self.b))
        else:
            self.a, self.b = W.random_bf16((self.M, self.K), seed), W.random_bf16(bsh, seed + 1)
            self.A.copy_(torch.from_numpy(self.a.view(np.int16))); self.B.copy_(torch.from_numpy(self.b.view(np.int16)))

    def call(self, stream):
        fn = G.gemm_s8s8_s32 if self.dtype == "int8" else G.gemm_bf16_f32acc_bf16
        ldb = self.N if self.layout == ROW else self.K
        return fn(self.M, self.N, self.K, self.A.data_ptr(), self.K, self.B.data_ptr(), ldb, self.layout,
                  self.C.data_ptr(), self.N, stream.cuda_stream)

    def check(self):
        C = self.C.cpu().numpy()
        if self.dtype == "int8":
            assert np.array_equal(C.astype(np.int64), oracle.gemm_s8(self.a, self.b, self.layout))
        else:
            ref, mag = oracle.gemm_bf16(self.a, self.b, self.layout)
            assert oracle.bf16_within_bound(C.view(np.uint16), ref, mag).all()


def test_graph_replay():
    G.gemm_reload_overrides()
    s = torch.cuda.Stream()
    jobs = [Job(*j) for j in JOBS]
    for i, j in enumerate(jobs):
        j.fill(i)
        assert j.call(s) == G.GEMM_OK  # warm-up outside capture: scratch of this stream grown
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for j in jobs:
            assert j.call(s) == G.GEMM_OK
    for rep in range(2):
        for i, j in enumerate(jobs):
            j.fill(100 * rep + 10 + i)
            j.C.zero_()
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        assert G.gemm_device_status() == G.GEMM_OK
        for j in jobs:
            j.check()
    # a larger call outside capture grows the stream's scratch; the graph's
    # buffers are kept, so it still replays correctly
    big = Job("int8", 1500, 2000, 3000, COL)
    big.fill(77)
    with torch.cuda.stream(s):
        assert big.call(s) == G.GEMM_OK
    torch.cuda.synchronize()
    big.check()
    for i, j in enumerate(jobs):
        j.fill(500 + i)
        j.C.zero_()
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    for j in jobs:
        j.check()


def test_capture_refuses_growth():
    G.gemm_reload_overrides()
    s = torch.cuda.Stream()
    small = Job("int8", 300, 400, 500, COL)
    small.fill(1)
    assert small.call(s) == G.GEMM_OK
    torch.cuda.synchronize()
    big = Job("int8", 2000, 2500, 3000, COL)  # needs more staging scratch than this stream has
    big.fill(2)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        assert big.call(s) == G.GEMM_ERR_UNSUPPORTED
        assert small.call(s) == G.GEMM_OK
    small.fill(3)
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    small.check()

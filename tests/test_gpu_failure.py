"""Failure detection on the GPU without faulting it: a bounded on-device
wait is made to run out (a barrier nothing arrives on), the kernel reports
GEMM_ERR_TIMEOUT through the device error word and returns normally, and the
context stays usable for further GEMMs."""
import numpy as np
import pytest
import torch

import oracle
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import workloads as W
from tests import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2512_13282_gb300 import build
    build.build()
    G.library()


def test_bounded_wait_expires_and_reports_timeout():
    assert G.gemm_device_status() == G.GEMM_OK
    assert G.gemm_selftest_wait_timeout(2_000_000) == G.GEMM_OK   # 2 ms
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_ERR_TIMEOUT
    assert G.gemm_device_status() == G.GEMM_OK                     # read clears it
    # the context is still usable
    A, B = W.random_int8((130, 300), 1), W.random_int8((300, 70), 2)
    C = U.run("int8", A, B, G.GEMM_B_ROW_MAJOR_KxN)
    assert np.array_equal(C.astype(np.int64), oracle.gemm_s8(A, B, oracle.B_ROW_MAJOR))


def test_selftest_rejects_unbounded_limits():
    assert G.gemm_selftest_wait_timeout(0) == G.GEMM_ERR_INVALID_ARG
    assert G.gemm_selftest_wait_timeout(2_000_000_000) == G.GEMM_ERR_INVALID_ARG

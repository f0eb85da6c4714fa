"""Host-side checks of the C ABI that need no GPU: the library builds for
sm_103a, loads, exports every function include/gb300_gemm.h declares, and
rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2512_13282_gb300 import build as B
from paper_2512_13282_gb300 import gemm as G

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = []
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            text = open(os.path.join(ROOT, "include", f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_ ]*?\**\s*\**\s*([a-z][a-z0-9_]*)\s*\(",
                                text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return G.library()


def test_exports_every_declared_symbol(lib):
    names = _declared_functions()
    assert "gemm_s8s8_s32" in names and "gemm_bf16_f32acc_bf16" in names
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"


def test_status_strings(lib):
    for s in range(5):
        assert G.gemm_status_string(s).startswith("GEMM_")
    assert "unknown" in G.gemm_status_string(99)


@pytest.mark.parametrize("fn", [G.gemm_s8s8_s32, G.gemm_bf16_f32acc_bf16])
def test_invalid_arguments_rejected_on_host(lib, fn):
    p = 0x1000  # never dereferenced: validation fails first
    bad = [
        (-1, 4, 4, p, 4, p, 4, 0, p, 4),        # negative M
        (4, 4, -2, p, 4, p, 4, 0, p, 4),        # negative K
        (4, 4, 4, p, 3, p, 4, 0, p, 4),         # lda < K
        (4, 5, 4, p, 4, p, 4, 0, p, 5),         # row-major ldb < N
        (4, 5, 6, p, 6, p, 5, 1, p, 5),         # column-major ldb < K
        (4, 5, 4, p, 4, p, 5, 0, p, 4),         # ldc < N
        (4, 4, 4, p, 4, p, 4, 2, p, 4),         # unknown layout
        (4, 4, 4, 0, 4, p, 4, 0, p, 4),         # null A
        (4, 4, 4, p, 4, 0, 4, 0, p, 4),         # null B
        (4, 4, 4, p, 4, p, 4, 0, 0, 4),         # null C
    ]
    for args in bad:
        assert fn(*args, stream=0) == G.GEMM_ERR_INVALID_ARG, args


@pytest.mark.parametrize("fn", [G.gemm_s8s8_s32, G.gemm_bf16_f32acc_bf16])
def test_empty_problems_are_noops(lib, fn):
    assert fn(0, 5, 7, 0, 7, 0, 5, 0, 0, 5, stream=0) == G.GEMM_OK
    assert fn(5, 0, 7, 0, 7, 0, 1, 0, 0, 1, stream=0) == G.GEMM_OK


@pytest.mark.parametrize("fn", [G.gemm_s8s8_s16, G.gemm_s8s8_s8])
def test_requantised_outputs_argument_checks_on_host(lib, fn):
    p = 0x1000
    for shift in (-1, 32, 100):
        assert fn(4, 4, 4, p, 4, p, 4, 0, p, 4, shift, stream=0) == G.GEMM_ERR_INVALID_ARG
    assert fn(4, 5, 4, p, 4, p, 5, 0, p, 4, 3, stream=0) == G.GEMM_ERR_INVALID_ARG  # ldc < N
    assert fn(4, 4, 4, p, 4, p, 4, 0, 0, 4, 3, stream=0) == G.GEMM_ERR_INVALID_ARG  # null C
    assert fn(0, 5, 7, 0, 7, 0, 5, 0, 0, 5, 31, stream=0) == G.GEMM_OK
    assert fn(2, 2, 131072, p, 131072, p, 2, 0, p, 2, 0, stream=0) == G.GEMM_ERR_UNSUPPORTED


def test_int8_k_limit_on_host(lib):
    p = 0x1000
    assert G.gemm_s8s8_s32(2, 2, 131072, p, 131072, p, 2, 0, p, 2, stream=0) == G.GEMM_ERR_UNSUPPORTED


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(G, "_lib", None)
    monkeypatch.setattr(G, "LIB_PATH", str(tmp_path / "nope.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        G.library()

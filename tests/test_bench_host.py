"""Host-side logic of the benchmark (no GPU): compulsory bytes and bound of a
GEMM, and the per-kernel-family lookup of recorded DRAM traffic."""
import json
import os

import pytest

import bench
from paper_2512_13282_gb300 import workloads as W


def _gemm(M, N, K, dtype):
    d = W.Dist("bf16") if dtype == "bf16" else W.Dist("int8")
    return W.Gemm(M, N, K, dtype, W.B_COL_MAJOR, 0, d, d)


def test_compulsory_bytes_and_bound():
    # A, B once each, C once: int8 inputs are 1 byte, int32 C 4; bf16 2 and 2
    assert bench.compulsory_bytes(_gemm(128, 256, 64, "int8")) == 128 * 64 + 64 * 256 + 128 * 256 * 4
    assert bench.compulsory_bytes(_gemm(128, 256, 64, "bf16")) == (128 * 64 + 64 * 256 + 128 * 256) * 2
    assert bench.compulsory_bytes(_gemm(8, 8, 8, "int8_int8")) == 8 * 8 + 8 * 8 + 8 * 8
    # 8192^3 bf16 is tensor-bound at the measured peaks, a GEMV is memory-bound
    assert bench.bound_of(_gemm(8192, 8192, 8192, "bf16"), 1950.0, 6693.8) == "tensor"
    assert bench.bound_of(_gemm(1, 11008, 4096, "bf16"), 1950.0, 6693.8) == "hbm"


def test_kernel_families_cover_existing_sources():
    for fam, files in bench.KERNEL_FAMILIES.items():
        for f in files:
            assert os.path.exists(os.path.join(bench.ROOT, "paper_2512_13282_gb300", "csrc", f)), (fam, f)
        assert len(bench.kernel_source_hash(fam)) == 16


def test_traffic_reported_only_for_the_recorded_sources(monkeypatch):
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    entries = rec["dram_bytes_per_launch"]
    assert entries, "no recorded traffic"
    name, e = next(iter(entries.items()))
    recorded = rec["kernel_source_hash"][e["family"]]
    monkeypatch.setattr(bench, "kernel_source_hash", lambda family="tc": recorded)
    assert bench.load_traffic(name) == e["bytes"]
    assert bench.load_traffic("no_such_gemm") is None
    monkeypatch.setattr(bench, "kernel_source_hash", lambda family="tc": "0" * 16)
    assert bench.load_traffic(name) is None


@pytest.mark.parametrize("fam", sorted(bench.KERNEL_FAMILIES))
def test_recorded_traffic_families_are_known(fam):
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    for e in rec["dram_bytes_per_launch"].values():
        assert e["family"] in bench.KERNEL_FAMILIES
        assert e["bytes"] > 0


def test_parse_shape():
    g = bench.parse_shape("int8:5120x4096x3000:row")
    assert (g.M, g.N, g.K, g.dtype, g.layout) == (5120, 4096, 3000, "int8", 0)
    g = bench.parse_shape("bf16:1x2x3:col")
    assert g.dtype == "bf16" and g.layout == 1
    for bad in ("int4:1x1x1:row", "int8:1x1:row", "int8:1x1x1:diag", "int8:0x1x1:row"):
        with pytest.raises(SystemExit):
            bench.parse_shape(bad)

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


import pytest  # noqa: E402


@pytest.fixture(autouse=True)
def _planner_overrides_follow_the_environment():
    """The library reads its GB300_GEMM_* planner overrides once; after each
    test (and after monkeypatch has restored the environment) they are read
    again, so that no test runs under another test's overrides."""
    yield
    from paper_2512_13282_gb300 import gemm as G
    if G._lib is not None:
        G.gemm_reload_overrides()

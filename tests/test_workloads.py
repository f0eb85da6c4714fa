"""The synthetic workloads (CPU): shapes, layouts, seeds and value
distributions of the five benchmark configurations, and the input recipe
(a fresh generator per GEMM, A drawn before B)."""
import numpy as np
import torch

from paper_2512_13282_gb300 import workloads as W


def _shapes(wl, dtype=None):
    return [(g.M, g.N, g.K) for g in W.WORKLOADS[wl].gemms if dtype is None or g.dtype == dtype]


def test_configurations():
    g256 = W.WORKLOADS["int8_square_256"].gemms
    assert [(g.M, g.N, g.K, g.dtype, g.layout, g.seed) for g in g256] == [(256, 256, 256, "int8", W.B_ROW_MAJOR, 0)]
    sweep = W.WORKLOADS["square_sweep_512_4096"].gemms
    assert sorted({(g.M, g.dtype) for g in sweep}) == sorted((s, d) for s in (512, 1024, 2048, 4096)
                                                            for d in ("int8", "bf16"))
    assert all(g.M == g.N == g.K and g.layout == W.B_COL_MAJOR and g.seed == 1 for g in sweep)
    big = W.WORKLOADS["square_8192"].gemms
    assert {(g.M, g.N, g.K, g.layout, g.seed) for g in big} == {(8192, 8192, 8192, W.B_ROW_MAJOR, 2)}
    assert all(g.a.scale == g.b.scale == 0.1 for g in big if g.dtype == "bf16")
    proj = W.WORKLOADS["transformer_projections"].gemms
    want = {(M, N, K) for M in (128, 2048) for (K, N) in ((4096, 4096), (4096, 11008), (11008, 4096), (4096, 12288))}
    assert set(_shapes("transformer_projections", "int8")) == want
    assert set(_shapes("transformer_projections", "bf16")) == want
    for g in proj:
        assert g.layout == W.B_COL_MAJOR and g.seed == 3
        if g.dtype == "int8":
            assert (g.a.lo, g.a.hi, g.b.lo, g.b.hi) == (-128, 127, -64, 63)
        else:
            assert (g.a.scale, g.b.scale) == (1.0, 0.02)
    irr = W.WORKLOADS["irregular_skinny"].gemms
    assert set(_shapes("irregular_skinny")) == {(1000, 1500, 3000), (16, 4096, 4096), (1, 11008, 4096),
                                                (3072, 2560, 777), (8192, 64, 8192)}
    assert all(g.layout == W.B_ROW_MAJOR and g.seed == 4 for g in irr)


def test_inputs_follow_the_recipe():
    g = W.Gemm(5, 7, 9, "int8", W.B_COL_MAJOR, 11, W.I8, W.I8_HALF)
    A, B = W.make_inputs(g)
    assert A.shape == (5, 9) and B.shape == (7, 9) and A.dtype == np.int8
    gen = torch.Generator().manual_seed(11)  # A first, then B, from one fresh generator
    assert np.array_equal(A, torch.randint(-128, 128, (5, 9), generator=gen, dtype=torch.int8).numpy())
    assert np.array_equal(B, torch.randint(-64, 64, (7, 9), generator=gen, dtype=torch.int8).numpy())
    A2, B2 = W.make_inputs(g)
    assert np.array_equal(A, A2) and np.array_equal(B, B2)
    gb = W.Gemm(64, 32, 48, "bf16", W.B_ROW_MAJOR, 2, W.BF, W.BF_002)
    A, B = W.make_inputs(gb)
    assert A.shape == (64, 48) and B.shape == (48, 32) and A.dtype == np.uint16
    a = (A.astype(np.uint32) << 16).view(np.float32)
    b = (B.astype(np.uint32) << 16).view(np.float32)
    assert np.isfinite(a).all() and np.isfinite(b).all()
    assert 0.5 < a.std() < 1.5 and 0.01 < b.std() < 0.03


def test_roofline_sweep_sizes():
    sizes = W.roofline_sweep_sizes()
    assert len(sizes) == 420 and len(set(sizes)) == 420
    assert all(256 <= x <= 8192 and x % 256 == 0 for t in sizes for x in t)

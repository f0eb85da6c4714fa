"""GPU parity: the CUDA library against the CPU oracle, element by element.

int8 results must equal the oracle's exact sums bit for bit; bf16 results
must satisfy |C - ref| <= 2^-8 |ref| + 2^-20 sum|a*b| for every element, and
equal the nearest-even rounding of the exact sum bit for bit whenever the
inputs make fp32 accumulation exact (integer-valued inputs).
"""
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


def _inputs(dtype, M, N, K, layout, seed):
    bshape = (K, N) if layout == ROW else (N, K)
    if dtype == "int8":
        return W.random_int8((M, K), seed), W.random_int8(bshape, seed + 1)
    return W.random_bf16((M, K), seed), W.random_bf16(bshape, seed + 1)


def _check(dtype, A, B, layout, C):
    if dtype == "int8":
        want = oracle.gemm_s8(A, B, layout)
        assert np.abs(want).max(initial=0) < 2 ** 31
        bad = np.argwhere(C.astype(np.int64) != want)
        assert bad.size == 0, f"{len(bad)} mismatches, first at {bad[:5].tolist()}: " \
                              f"{C[tuple(bad[0])]} vs {want[tuple(bad[0])]}"
    else:
        ref, mag = oracle.gemm_bf16(A, B, layout)
        ok = oracle.bf16_within_bound(C, ref, mag)
        bad = np.argwhere(~ok)
        assert bad.size == 0, f"{len(bad)} out of bound, first at {bad[:5].tolist()}"
        _check_rounding(C, ref)


def _bf16_order(bits):
    """bf16 bit patterns as integers in the order of their values (adjacent
    representable values differ by 1)."""
    b = bits.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def _check_rounding(C, ref):
    """With fp32 accumulation and one rounding, nearly every element is the
    correctly rounded exact sum and the rest are one bf16 step from it (sums
    that lie within the fp32 error of a rounding boundary, or cancel to far
    below their terms).  A kernel that truncated, rounded twice or dropped a
    term would leave many elements one step off or more."""
    want = oracle.rne_bf16(ref)
    fin = np.isfinite(ref) & np.isfinite(oracle.bf16_bits_to_f64(C))
    if not fin.any():
        return
    steps = np.abs(_bf16_order(C[fin]) - _bf16_order(want[fin]))
    exact = np.mean(steps == 0)
    far = np.mean(steps > 1)
    assert exact >= 0.95, f"only {exact:.4f} of elements are the correctly rounded sum"
    assert far <= 0.005, f"{far:.4f} of elements are more than one bf16 step from the correctly rounded sum"


SHAPES = [
    (1, 1, 1), (5, 7, 3), (128, 256, 64), (129, 257, 65), (300, 520, 200),
    (64, 1000, 1100), (257, 129, 2100), (130, 700, 4096), (1000, 1500, 3000),
]


@pytest.mark.parametrize("dtype", ["int8", "bf16", "int8-tensor"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", SHAPES, ids=[f"{m}x{n}x{k}" for m, n, k in SHAPES])
def test_parity_shapes(dtype, layout, M, N, K, monkeypatch):
    """As routed by the planner (int8 problems this small run in one launch
    on the CUDA cores), and int8 on the tensor-core kernels (forced)."""
    if dtype == "int8-tensor":
        dtype = "int8"
        monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    A, B = _inputs(dtype, M, N, K, layout, seed=M * 7 + N * 3 + K)
    C = U.run(dtype, A, B, layout)
    _check(dtype, A, B, layout, C)


SPLITK = [(16, 512, 4096), (128, 256, 8192), (1, 300, 5000), (3, 64, 20000)]


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", SPLITK, ids=[f"{m}x{n}x{k}" for m, n, k in SPLITK])
def test_parity_split_k(dtype, layout, M, N, K):
    A, B = _inputs(dtype, M, N, K, layout, seed=11)
    C = U.run(dtype, A, B, layout)
    _check(dtype, A, B, layout, C)


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("pads", [(1, 3, 5, 0, 0, 0), (0, 0, 0, 1, 1, 1), (8, 8, 8, 8, 8, 8),
                                  (3, 0, 1, 0, 5, 3)],
                         ids=["odd_ld", "odd_base", "wide_ld", "mixed"])
def test_parity_leading_dims_and_offsets(dtype, layout, pads):
    M, N, K = 200, 333, 777
    pa, pb, pc, oa, ob, oc = pads
    A, B = _inputs(dtype, M, N, K, layout, seed=21)
    bcols = N if layout == ROW else K
    C = U.run(dtype, A, B, layout, lda=K + pa, ldb=bcols + pb, ldc=N + pc, a_off=oa, b_off=ob, c_off=oc)
    _check(dtype, A, B, layout, C)


@pytest.mark.parametrize("dtype", ["int8", "bf16", "int8_int16", "int8_int8"])
@pytest.mark.parametrize("pair", ["0", "1"], ids=["single", "pair"])
@pytest.mark.parametrize("N", [333, 5])
def test_row_ends_inside_padded_pitch(dtype, pair, N, monkeypatch):
    """C rows whose pitch is a multiple of 16 bytes but whose last element
    is not at a 16-byte boundary (ldc > N): nothing of the padding between
    column N and the pitch may be written (a TMA store clipped at N still
    writes the rest of the row's last 16-byte piece, so such C is stored
    directly).  The guard check of U.run covers the padding."""
    monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    monkeypatch.setenv("GB300_GEMM_PAIR", pair)
    M, K = 300, 777
    esize = {"int8": 4, "bf16": 2, "int8_int16": 2, "int8_int8": 1}[dtype]
    ldc = N + 1
    while (ldc * esize) % 16:
        ldc += 1
    assert (N * esize) % 16 != 0
    base = "bf16" if dtype == "bf16" else "int8"
    A, B = _inputs(base, M, N, K, COL, seed=N + len(dtype))
    shift = 9 if dtype in ("int8_int16", "int8_int8") else 0
    C = U.run(dtype, A, B, COL, ldc=ldc, shift=shift)
    if dtype in ("int8", "bf16"):
        _check(dtype, A, B, COL, C)
    else:
        want = oracle.requantize(oracle.gemm_s8(A, B, COL), shift, 16 if dtype == "int8_int16" else 8)
        assert np.array_equal(C.astype(np.int64), want)


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
def test_bf16_integer_inputs_bit_exact(layout):
    """Integer-valued inputs in [-8, 8]: fp32 accumulation is exact in any
    order, so C must be the correctly rounded exact sum, bit for bit."""
    M, N, K = 300, 400, 1500
    A = W.integer_bf16((M, K), 31)
    B = W.integer_bf16((K, N) if layout == ROW else (N, K), 32)
    C = U.run("bf16", A, B, layout)
    ref, _ = oracle.gemm_bf16(A, B, layout)
    assert np.array_equal(C, oracle.rne_bf16(ref))


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
def test_int8_all_minus128(layout):
    """All -128: every 1024-long slab sums to exactly 2^24."""
    M, N, K = 130, 260, 4096
    A = np.full((M, K), -128, np.int8)
    B = np.full((K, N) if layout == ROW else (N, K), -128, np.int8)
    C = U.run("int8", A, B, layout)
    assert (C == 16384 * K).all()


def test_int8_edge_of_fp32_exactness():
    """Slab sums of 1023 * 2^14 + 1 = 16760833: odd and just below 2^24, so
    every bit of the fp32 significand is needed; signs vary by column."""
    M, N, K = 128, 256, 3072
    A = np.full((M, K), -128, np.int8)
    A[:, 1023::1024] = 1
    B = np.full((K, N), -128, np.int8)
    B[1023::1024, :] = 1
    sign = np.where(np.arange(N) % 3 == 0, -1, 1)
    B = (B.astype(np.int16) * sign[None, :]).clip(-128, 127).astype(np.int8)
    C = U.run("int8", A, B, ROW)
    _check("int8", A, B, ROW, C)


def test_int8_largest_exact_k():
    """K = 131071 with all -128 gives 2147467264, the largest int32 the
    exactness rule admits (split-K and slabs both involved)."""
    M, N, K = 3, 5, 131071
    A = np.full((M, K), -128, np.int8)
    B = np.full((N, K), -128, np.int8)
    C = U.run("int8", A, B, COL)
    assert (C == 2147467264).all()
    B2 = np.full((N, K), 127, np.int8)
    C2 = U.run("int8", A, B2, COL)
    assert (C2 == -16256 * K).all()


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
def test_k_zero_writes_zeros(dtype):
    M, N = 70, 90
    A = np.zeros((M, 0), np.int8 if dtype == "int8" else np.uint16)
    B = np.zeros((0, N), A.dtype)
    C = U.run(dtype, A, B, ROW)
    assert (C == 0).all()


def test_bf16_special_values():
    M, N, K = 4, 300, 200
    A = W.random_bf16((M, K), 41)
    B = np.abs(W.random_bf16((K, N), 42).view(np.int16)).view(np.uint16)  # clear sign bits
    A[0, 0] = 0x7FC0   # NaN
    A[1, 5] = 0x7F80   # +inf
    A[2, 7] = 0xFF80   # -inf
    C = U.run("bf16", A, B, ROW)
    _check("bf16", A, B, ROW, C)
    c = oracle.bf16_bits_to_f64(C)
    assert np.isnan(c[0]).all() and np.isposinf(c[1]).all() and np.isneginf(c[2]).all()


def test_int8_k_too_large_rejected():
    A = np.zeros((2, 131072), np.int8)
    B = np.zeros((131072, 2), np.int8)
    U.run("int8", A, B, ROW, expect=G.GEMM_ERR_UNSUPPORTED)


def test_workspace_reuse_and_streams():
    """Back-to-back calls of different sizes on a side stream reuse and grow
    the workspace; results stay exact."""
    s = torch.cuda.Stream()
    for (M, N, K) in ((16, 512, 4096), (1, 3000, 9000), (300, 200, 100), (16, 512, 4096)):
        A, B = _inputs("int8", M, N, K, COL, seed=M + N)
        C = U.run("int8", A, B, COL, stream=s)
        _check("int8", A, B, COL, C)


def test_launch_counter_advances():
    before = G.gemm_launch_count()
    A, B = _inputs("bf16", 64, 64, 64, ROW, seed=5)
    U.run("bf16", A, B, ROW)
    assert G.gemm_launch_count() > before


# ------------------------------------------------ full-size configurations

def _sample_positions(M, N, BN=128, BMt=128, cap=12000, seed=0):
    """Tile corners and edges (tiles of BMt rows x BN columns, plus the
    128-row and 128-column grid) and random interior points."""
    rng = np.random.default_rng(seed)
    rows = set()
    for step in {128, BMt}:
        for r0 in range(0, M, step):
            rows.update({r0, min(r0 + step - 1, M - 1)})
    cols = set()
    for step in {128, BN}:
        for c0 in range(0, N, step):
            cols.update({c0, min(c0 + step - 1, N - 1)})
    rows, cols = np.array(sorted(rows)), np.array(sorted(cols))
    rr, cc = np.meshgrid(rows, cols, indexing="ij")
    r = np.concatenate([rr.ravel(), rng.integers(0, M, cap // 2), [M - 1]])
    c = np.concatenate([cc.ravel(), rng.integers(0, N, cap // 2), [N - 1]])
    if r.size > cap:
        keep = rng.choice(r.size, cap, replace=False)
        r, c = r[keep], c[keep]
    return r.astype(np.int64), c.astype(np.int64)


WHOLE = [g for w in ("int8_square_256", "square_sweep_512_4096", "irregular_skinny") for g in W.WORKLOADS[w].gemms]


@pytest.mark.parametrize("g", WHOLE, ids=[g.name for g in WHOLE])
def test_full_size_configs_whole(g):
    """The 256^3, square sweep (512^3 .. 4096^3, both paths) and irregular /
    skinny GEMMs at full size, in the launch configuration the benchmark
    times: every element against the oracle (int8 bit for bit, bf16 within
    the bound and correctly rounded)."""
    A, B = W.make_inputs(g)
    C = U.run(g.dtype, A, B, g.layout, shift=g.shift)
    _check(g.dtype, A, B, g.layout, C)


def _plan_tiles(g):
    """(rows, columns) of the output tiles the planner uses for g."""
    st, plan = G.gemm_plan_query(g.M, g.N, g.K, g.int8_in, g.layout)
    assert st == 0
    if plan["route"] == G.GEMM_ROUTE_TC_PAIR:
        return 256, plan["bn"]
    if plan["route"] == G.GEMM_ROUTE_TC_SINGLE:
        return 128, plan["bn"]
    return 128, 128


SAMPLED = [g for w in ("square_8192", "transformer_projections", "reduced_precision_outputs")
           for g in W.WORKLOADS[w].gemms]


@pytest.mark.parametrize("g", SAMPLED, ids=[g.name for g in SAMPLED])
def test_full_size_configs_sampled(g):
    """The 8192^3, transformer projection and reduced-precision GEMMs at full
    size, in the launch configuration the benchmark times: outputs at the
    corners and edges of the tiles the planner chose (e.g. 224 columns, 256
    rows per CTA pair) and at random points, against the oracle one by one."""
    A, B = W.make_inputs(g)
    C = U.run(g.dtype, A, B, g.layout, shift=g.shift)
    bm, bn = _plan_tiles(g)
    r, c = _sample_positions(g.M, g.N, BN=bn, BMt=bm, seed=g.M + g.N + g.K)
    if g.int8_in:
        want = oracle.gemm_s8_entries(A, B, g.layout, r, c)
        if g.dtype != "int8":
            want = oracle.requantize(want, g.shift, 8 * g.out_bytes)
        got = C[r, c].astype(np.int64)
        assert np.array_equal(got, want), f"{np.sum(got != want)} of {r.size} sampled entries differ"
    else:
        ref, mag = oracle.gemm_bf16_entries(A, B, g.layout, r, c)
        assert oracle.bf16_within_bound(C[r, c], ref, mag).all()
        _check_rounding(C[r, c], ref)


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("bn", [128, 192, 224, 256])
@pytest.mark.parametrize("pair", ["0", "1"], ids=["single", "pair"])
def test_parity_every_tile_width(dtype, layout, bn, pair, monkeypatch):
    """Each compiled kernel family (one CTA per 128-row tile, or CTA pairs
    per 256-row tile) and tile width -- the planner normally picks one per
    shape -- on ragged multi-tile shapes, with and without split-K."""
    monkeypatch.setenv("GB300_GEMM_BN", str(bn))
    monkeypatch.setenv("GB300_GEMM_PAIR", pair)
    for (M, N, K, splits) in ((300, 700, 1500, "1"), (130, 450, 3000, "3")):
        monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
        A, B = _inputs(dtype, M, N, K, layout, seed=bn + M)
        C = U.run(dtype, A, B, layout)
        _check(dtype, A, B, layout, C)


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("bn", [64, 96])
def test_parity_narrow_bf16_tiles(layout, bn, monkeypatch):
    """The 64- and 96-wide bf16 kernels (96 for B column-major only) on
    ragged multi-tile shapes, N narrower than one tile, few rows and long K,
    with and without split-K; the plan query reports the forced width."""
    if layout == ROW and bn == 96:
        pytest.skip("no 96-wide tile for row-major B")
    monkeypatch.setenv("GB300_GEMM_BN", str(bn))
    monkeypatch.setenv("GB300_GEMM_PAIR", "0")
    for (M, N, K, splits) in ((300, 700, 1500, "1"), (130, 450, 3000, "3"), (128, 1100, 2048, "1"),
                              (1000, 64, 4100, "2"), (129, 97, 333, "1"), (40, 200, 5000, "4")):
        monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
        G.gemm_reload_overrides()
        st, plan = G.gemm_plan_query(M, N, K, False, layout)
        assert st == 0 and plan["route"] == G.GEMM_ROUTE_TC_SINGLE and plan["bn"] == bn, plan
        A, B = _inputs("bf16", M, N, K, layout, seed=bn + M + N)
        C = U.run("bf16", A, B, layout)
        _check("bf16", A, B, layout, C)


SPLIT_TAIL = [  # (M, N, K, BN, pair, T): 165 = 152 + 13 tiles, 81 = 76 + 5 pairs
    (1300, 1900, 777, 128, "0", 2), (1300, 1901, 2500, 128, "0", 3),
    (2100, 2300, 1000, 256, "1", 2), (2100, 2303, 2500, 256, "1", 4),
]


@pytest.mark.parametrize("dtype", ["int8", "bf16", "int8_int16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K,bn,pair,T", SPLIT_TAIL,
                         ids=[f"{m}x{n}x{k}-bn{b}-{'pair' if p == '1' else 'single'}-T{t}"
                              for m, n, k, b, p, t in SPLIT_TAIL])
def test_parity_split_tail(dtype, layout, M, N, K, bn, pair, T, monkeypatch):
    """Split tail: the tiles of the last, partly filled round are split in T
    K ranges (crossing int8 1024-deep slabs) that write partials, reduced
    over those tiles only, while every other tile writes C -- ragged edges,
    N with rows not ending on a 16-byte boundary (partials stored directly),
    TMA and direct stores (GB300_GEMM_TMA_STORE=0), int16 requantisation;
    the plan query reports the split tail."""
    monkeypatch.setenv("GB300_GEMM_BN", str(bn))
    monkeypatch.setenv("GB300_GEMM_PAIR", pair)
    monkeypatch.setenv("GB300_GEMM_TAIL_SPLITS", str(T))
    G.gemm_reload_overrides()
    st, plan = G.gemm_plan_query(M, N, K, dtype != "bf16", layout)
    assert st == 0 and plan["tail_splits"] == T and plan["splits"] == 1 and plan["bn"] == bn, plan
    src = "bf16" if dtype == "bf16" else "int8"
    A, B = _inputs(src, M, N, K, layout, seed=M + N + K + T)
    for tma in ("1", "0"):
        monkeypatch.setenv("GB300_GEMM_TMA_STORE", tma)
        if dtype == "int8_int16":
            C = U.run(dtype, A, B, layout, shift=5)
            assert np.array_equal(C.astype(np.int64), oracle.requantize(oracle.gemm_s8(A, B, layout), 5, 16))
        else:
            _check(src, A, B, layout, U.run(dtype, A, B, layout))


SKINNY = [(1, 1, 1), (1, 11008, 4096), (2, 257, 777), (3, 1000, 4100), (5, 300, 64), (8, 4096, 4096),
          (13, 555, 2049), (16, 4096, 4096), (16, 96, 20000)]


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", SKINNY, ids=[f"{m}x{n}x{k}" for m, n, k in SKINNY])
@pytest.mark.parametrize("path", ["auto", "cudacore", "tensor"])
def test_parity_small_m(dtype, layout, M, N, K, path, monkeypatch):
    """M <= 16: the CUDA-core small-M kernel (forced, or as the planner
    routes it) and the tensor-core path (forced), full comparison."""
    if path == "cudacore":
        monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "16")
    elif path == "tensor":
        monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    A, B = _inputs(dtype, M, N, K, layout, seed=M * 31 + N)
    C = U.run(dtype, A, B, layout)
    _check(dtype, A, B, layout, C)


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
def test_small_m_misaligned_and_repeated(dtype, layout, monkeypatch):
    """Odd leading dimensions and bases take the scalar load paths; calls in
    a row reuse the self-resetting reduction counters."""
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "16")
    for rep, (M, N, K) in enumerate(((7, 333, 3001), (16, 1024, 8192), (7, 333, 3001))):
        A, B = _inputs(dtype, M, N, K, layout, seed=rep)
        bcols = N if layout == ROW else K
        C = U.run(dtype, A, B, layout, lda=K + 3, ldb=bcols + 1, ldc=N + 2, a_off=1, b_off=3, c_off=1)
        _check(dtype, A, B, layout, C)


@pytest.mark.parametrize("dtype", ["int8", "bf16"])
@pytest.mark.parametrize("M", [1, 2, 4, 8, 16])
def test_small_m_row_b_alignments(dtype, M, monkeypatch):
    """Row-major B whose base and row pitch are aligned to 16, 8, 4, 2 and 1
    bytes: the small-M kernel loads 16, 8 or 4 bytes of a row per lane where
    the alignment allows, else element by element; N ragged against every
    lane width and K against the kernel's row batches."""
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "16")
    esize = 1 if dtype == "int8" else 2
    N, K = 1000, 1234
    for align in (16, 8, 4, 2, 1):
        if align < esize:
            continue
        el = align // esize  # elements of the alignment
        ldb = -(-N // el) * el  # a pitch aligned to exactly `align` bytes (at least 16 for 16)
        if align < 16 and (ldb * esize) % (2 * align) == 0:
            ldb += el
        b_off = 0 if align == 16 else el
        A, B = _inputs(dtype, M, N, K, ROW, seed=align * 7 + M)
        C = U.run(dtype, A, B, ROW, ldb=ldb, b_off=b_off)
        _check(dtype, A, B, ROW, C)


def test_small_m_int8_extremes(monkeypatch):
    """dp4a exactness at the int32 edge: K = 131071 of (-128)(-128)."""
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "16")
    for layout in (ROW, COL):
        M, N, K = 2, 40, 131071
        A = np.full((M, K), -128, np.int8)
        B = np.full((K, N) if layout == ROW else (N, K), -128, np.int8)
        C = U.run("int8", A, B, layout)
        assert (C == 2147467264).all()


# ------------------------------------- int8 problems in one CUDA-core launch

TINY = [(1, 1, 1), (9, 33, 65), (33, 65, 77), (256, 256, 256), (512, 512, 512), (200, 300, 500), (100, 700, 1001),
        (40, 50, 6000)]


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", TINY, ids=[f"{m}x{n}x{k}" for m, n, k in TINY])
def test_int8_tiny_problems(layout, M, N, K, monkeypatch):
    """Small int8 problems in one launch of the CUDA-core tile kernel (dp4a,
    row-major B byte-transposed on the fly): ragged 32 x 32 tiles and K
    chunks, bit-exact against the oracle."""
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    G.gemm_reload_overrides()
    A, B = _inputs("int8", M, N, K, layout, seed=M + 3 * N + K)
    st, plan = G.gemm_plan_query(M, N, K, True, layout)
    assert plan["route"] == G.GEMM_ROUTE_TINY
    C = U.run("int8", A, B, layout)
    _check("int8", A, B, layout, C)


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
def test_int8_tiny_kernel_forced_misaligned_and_extreme(layout, monkeypatch):
    """Forced onto larger and misaligned problems: odd leading dimensions and
    bases (scalar loads), requantised outputs, and K = 131071 of all -128."""
    monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", str(1 << 40))
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    M, N, K = 300, 333, 2049
    A, B = _inputs("int8", M, N, K, layout, seed=5)
    bcols = N if layout == ROW else K
    C = U.run("int8", A, B, layout, lda=K + 3, ldb=bcols + 1, ldc=N + 2, a_off=1, b_off=3, c_off=1)
    _check("int8", A, B, layout, C)
    for out, shift in (("int8_int16", 9), ("int8_int8", 17)):
        C = U.run(out, A, B, layout, shift=shift)
        want = oracle.requantize(oracle.gemm_s8(A, B, layout), shift, 16 if out == "int8_int16" else 8)
        assert np.array_equal(C.astype(np.int64), want)
    A = np.full((40, 131071), -128, np.int8)
    B = np.full((131071, 48) if layout == ROW else (48, 131071), -128, np.int8)
    assert (U.run("int8", A, B, layout) == 2147467264).all()


# ------------------------------------------- int8 operand staging variants

STAGING = [(300, 520, 256), (1000, 1500, 3000), (257, 129, 4096), (640, 2048, 784), (2048, 2048, 2048),
           (200, 300, 775)]


@pytest.mark.parametrize("layout", [ROW, COL], ids=["Brow", "Bcol"])
@pytest.mark.parametrize("M,N,K", STAGING, ids=[f"{m}x{n}x{k}" for m, n, k in STAGING])
@pytest.mark.parametrize("pdl", ["1", "0"], ids=["pdl", "nopdl"])
def test_int8_staging_with_and_without_programmatic_launch(layout, M, N, K, pdl, monkeypatch):
    """The staging pass (flat vectors for tight operands, per-row chunks
    otherwise) followed by the GEMM, launched with and without programmatic
    dependent launch: bit-exact either way."""
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    monkeypatch.setenv("GB300_GEMM_TINY_MAX_MACS", "0")
    monkeypatch.setenv("GB300_GEMM_PDL", pdl)
    A, B = _inputs("int8", M, N, K, layout, seed=M ^ N ^ K)
    C = U.run("int8", A, B, layout)
    _check("int8", A, B, layout, C)


def test_int8_back_to_back_calls(monkeypatch):
    """Calls queued back to back on one stream without synchronising (pairs,
    split-K and its reduction included) share the staging workspace: each
    GEMM must read its own staged operands, never the next call's."""
    seq = [(2048, 1024, 4096, COL, "1", None), (512, 512, 512, ROW, "0", None),
           (130, 700, 8192, COL, "0", "4"), (1024, 2048, 1024, ROW, "1", None), (2048, 1024, 4096, COL, "1", None)]
    keep = []
    for M, N, K, layout, pair, splits in seq:
        monkeypatch.setenv("GB300_GEMM_PAIR", pair)
        if splits:
            monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
        else:
            monkeypatch.delenv("GB300_GEMM_SPLITS", raising=False)
        A, B = _inputs("int8", M, N, K, layout, seed=K + M)
        abuf, pa, lda = U.to_device(A)
        bbuf, pb, ldb = U.to_device(B)
        C = torch.empty((M, N), dtype=torch.int32, device="cuda")
        G.gemm_reload_overrides()
        assert G.gemm_s8s8_s32(M, N, K, pa, lda, pb, ldb, layout, C, N) == G.GEMM_OK
        keep.append((A, B, layout, abuf, bbuf, C))
    torch.cuda.synchronize()
    assert G.gemm_device_status() == G.GEMM_OK
    for A, B, layout, _, _, C in keep:
        _check("int8", A, B, layout, C.cpu().numpy())


# ------------------------ int8 with the large operand converted in the kernel

S8TM = [
    # M <= 128, B stored N x K: the weights are streamed as int8 (swap)
    (16, 512, 4096, COL), (128, 4096, 1000, COL), (100, 1000, 3000, COL), (64, 300, 64, COL),
    (9, 129, 1024, COL), (128, 1500, 8192, COL),
    # M <= 128, B stored K x N (N a multiple of 16, so its rows are TMA-legal):
    # the weights are streamed as int8 and read transposed by the converters
    (16, 512, 4096, ROW), (128, 4096, 1000, ROW), (100, 1008, 3000, ROW), (64, 304, 64, ROW),
    (9, 144, 1024, ROW), (128, 1520, 8192, ROW), (17, 160, 1000, ROW),
    # N <= 128, M > 128: A is streamed as int8, B (either layout) staged
    (1000, 64, 3008, ROW), (300, 128, 4096, COL), (2000, 17, 1024, ROW), (129, 100, 2048, COL),
    (640, 65, 11008, ROW),
]


@pytest.mark.parametrize("M,N,K,layout", S8TM, ids=[f"{m}x{n}x{k}-{'Bcol' if l else 'Brow'}"
                                                    for m, n, k, l in S8TM])
@pytest.mark.parametrize("splits", ["auto", "1", "3"])
def test_int8_converted_in_kernel(M, N, K, layout, splits, monkeypatch):
    """The int8 kernel that converts its large operand to bf16 in tensor
    memory (swap for small M, with B read K-major or transposed; direct for
    small N): ragged tiles in every dimension, forced split-K, bit-exact
    against the oracle."""
    if splits != "auto":
        monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
    A, B = _inputs("int8", M, N, K, layout, seed=M * 5 + N + K)
    C = U.run("int8", A, B, layout)
    _check("int8", A, B, layout, C)


@pytest.mark.parametrize("M,N,K,layout", [(16, 512, 4096, COL), (16, 512, 4096, ROW), (300, 128, 4096, ROW)],
                         ids=["swap", "swap-transposed", "direct"])
@pytest.mark.parametrize("out", ["int8_int16", "int8_int8"])
@pytest.mark.parametrize("shift", [0, 7, 12])
def test_int8_converted_in_kernel_requantised(M, N, K, layout, out, shift):
    A, B = _inputs("int8", M, N, K, layout, seed=shift + M)
    C = U.run(out, A, B, layout, shift=shift)
    want = oracle.requantize(oracle.gemm_s8(A, B, layout), shift, 16 if out == "int8_int16" else 8)
    assert np.array_equal(C.astype(np.int64), want)


def test_int8_converted_in_kernel_extremes(monkeypatch):
    """All -128 (every 1024-deep slab is exactly 2^24), the largest exact K,
    and M = 1 on this path (the CUDA-core kernel turned off)."""
    A = np.full((128, 4096), -128, np.int8)
    B = np.full((300, 4096), -128, np.int8)
    assert (U.run("int8", A, B, COL) == 16384 * 4096).all()
    A = np.full((16, 131071), -128, np.int8)
    B = np.full((200, 131071), -128, np.int8)
    assert (U.run("int8", A, B, COL) == 2147467264).all()
    B[:, :] = 127
    assert (U.run("int8", A, B, COL) == -16256 * 131071).all()
    monkeypatch.setenv("GB300_GEMM_SKINNY_MAX_M", "0")
    A1, B1 = _inputs("int8", 1, 700, 640, COL, seed=3)
    _check("int8", A1, B1, COL, U.run("int8", A1, B1, COL))
    # B stored K x N, read transposed: M = 1..8 (normally the CUDA-core
    # kernel's), all -128 and the largest exact K
    for M in (1, 2, 5, 8):
        A1, B1 = _inputs("int8", M, 272, 1100, ROW, seed=M)
        _check("int8", A1, B1, ROW, U.run("int8", A1, B1, ROW))
    A = np.full((16, 131071), -128, np.int8)
    B = np.full((131071, 160), -128, np.int8)
    assert (U.run("int8", A, B, ROW) == 2147467264).all()


@pytest.mark.parametrize("M,N,K,layout", [(128, 4096, 4096, COL), (128, 11008, 4096, COL), (16, 4096, 4096, ROW),
                                          (8192, 64, 8192, ROW)],
                         ids=["swap", "swap-wide", "swap-transposed", "direct"])
def test_int8_converted_in_kernel_matches_general_path(M, N, K, layout, monkeypatch):
    """Full-size shapes of the benchmark: the new path and the general
    (staged) path give the same int32 results, and sampled entries match the
    oracle."""
    A, B = _inputs("int8", M, N, K, layout, seed=7)
    C1 = U.run("int8", A, B, layout)
    monkeypatch.setenv("GB300_GEMM_S8TM", "0")
    C0 = U.run("int8", A, B, layout)
    assert np.array_equal(C0, C1)
    r, c = _sample_positions(M, N, seed=3)
    assert np.array_equal(C1[r, c].astype(np.int64), oracle.gemm_s8_entries(A, B, layout, r, c))


@pytest.mark.parametrize("M,N,K,layout", [(16, 512, 4096, COL), (100, 1000, 3000, COL), (1000, 64, 3008, ROW),
                                          (100, 1008, 3000, ROW)],
                         ids=["swap", "swap-ragged", "direct", "swap-transposed"])
@pytest.mark.parametrize("splits", ["3", "8"])
def test_int8_converted_in_kernel_split_into_padded_c(M, N, K, layout, splits, monkeypatch):
    """Split-K of int32 outputs on the small-operand path adds every split's
    exact partial sums into C, zeroed beforehand: C with a padded pitch and
    an offset base, nothing outside [0,M) x [0,N) written."""
    monkeypatch.setenv("GB300_GEMM_SPLITS", splits)
    A, B = _inputs("int8", M, N, K, layout, seed=M + K)
    C = U.run("int8", A, B, layout, ldc=N + 5, c_off=3)
    _check("int8", A, B, layout, C)


@pytest.mark.parametrize("M,N,K,layout", [(16, 512, 4096, COL), (100, 1008, 3000, ROW), (1000, 64, 3008, ROW),
                                          (300, 128, 4096, COL), (9, 144, 1024, ROW)],
                         ids=["swap", "swap-transposed", "direct", "direct-Bcol", "swap-small"])
@pytest.mark.parametrize("ldc_pad", [0, 4, 12])
def test_int8_converted_in_kernel_split_tma_reduction(M, N, K, layout, ldc_pad, monkeypatch):
    """Split-K of int32 outputs on the small-operand path where C allows TMA
    (16-byte aligned base and pitch, rows ending on a 16-byte boundary):
    the splits' sums go into C by TMA tensor reductions, clipped at the
    matrix edges (ragged tiles, padded pitch untouched), bit-exact and equal
    to the element-wise atomic adds (GB300_GEMM_TMA_STORE=0)."""
    monkeypatch.setenv("GB300_GEMM_SPLITS", "3")
    A, B = _inputs("int8", M, N, K, layout, seed=M + N + ldc_pad)
    C = U.run("int8", A, B, layout, ldc=N + ldc_pad)
    _check("int8", A, B, layout, C)
    monkeypatch.setenv("GB300_GEMM_TMA_STORE", "0")
    assert np.array_equal(U.run("int8", A, B, layout, ldc=N + ldc_pad), C)

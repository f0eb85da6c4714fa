"""The tile model and planner (the paper's Sec. 4.5, Eq. 1-10, restated for
GB300) on the CPU: the compiled kernels' pipeline depths are the deepest the
shared-memory budget allows (Eq. 5); the planner built into the library and
the Python model choose the same plan; the planner's cost table is the one
the model fits to the committed measurements; and on those measurements the
model's choices are close to the best forced plan."""
import json
import os
import random

import numpy as np
import pytest

from paper_2512_13282_gb300 import build as B
from paper_2512_13282_gb300 import gemm as G
from paper_2512_13282_gb300 import tile_model as T

OVERRIDES = ("GB300_GEMM_BN", "GB300_GEMM_PAIR", "GB300_GEMM_SPLITS", "GB300_GEMM_TAIL_SPLITS", "GB300_GEMM_SKINNY_MAX_M",
             "GB300_GEMM_S8TM", "GB300_GEMM_TMA_STORE", "GB300_GEMM_TINY_MAX_MACS")


@pytest.fixture()
def lib(monkeypatch):
    B.build()
    G.library()
    for k in OVERRIDES:
        monkeypatch.delenv(k, raising=False)
    G.gemm_reload_overrides()
    return G


def test_single_core_ip_prefers_the_largest_tile_that_fits():
    """Sec. 4.5.1 on one SM: most MACs per stage first, then the smallest
    output tile.  With the 128-byte swizzle capping BK at 64 and two fp32
    accumulators in 512 TMEM columns, that is 128 x 256 x 64 (single CTA)
    and 256 x 256 x 64 (CTA pair)."""
    best = T.single_core_ip()[0]
    assert (best["bm"], best["bn"], best["bk"]) == (128, 256, 64)
    assert best["comp_cycles"] >= best["comm_cycles"]          # Eq. 4
    best2 = T.single_core_ip(pair=True)[0]
    assert (best2["bm"], best2["bn"], best2["bk"]) == (256, 256, 64)
    # a tile too narrow for its TMA fill fails Eq. 4
    assert all(r["bn"] >= 64 for r in T.single_core_ip())


def test_every_compiled_variant_satisfies_eq4_and_eq5():
    """Eq. 5 (the ring fits) for every compiled kernel, Eq. 4 (a stage's
    MMA time covers its TMA fill) for all but the narrow bf16 tiles, which
    exist for memory-bound GEMMs and are chosen only by measured time."""
    for v in T.compiled_variants():
        comp, comm = v.eq4_cycles()
        assert (comp >= comm) == (v.bn not in T.NARROW), v
        s = v.max_stages()
        assert s >= 2 and v.smem_bytes(s) <= T.GB300["smem_per_cta"] < v.smem_bytes(s + 1), v
        assert v.tmem_cols() <= T.GB300["tmem_cols"], v


def test_planner_widths_are_the_compiled_variants():
    """The widths the planner may pick per operand type, family and B
    layout are exactly the compiled kernels."""
    compiled = {(v.dtype, v.pair, v.bn, km) for v in T.compiled_variants() for km in (True, False)
                if km or not v.kmajor_only}
    planned = {(d, pair, bn, km) for d in ("bf16", "int8") for pair in (False, True) for km in (True, False)
               for bn in T.plan_widths(d, pair, km)}
    assert planned == compiled


@pytest.mark.parametrize("dtype", ["bf16", "int8"])
@pytest.mark.parametrize("pair", [False, True], ids=["single", "pair"])
@pytest.mark.parametrize("bn", [64, 96, 128, 192, 224, 256])
def test_library_pipeline_depths_are_the_model_maximum(lib, monkeypatch, dtype, pair, bn):
    """The stage count the library compiles for each variant equals Eq. 5's
    maximum (the C++ derives it from the same budget)."""
    if bn in T.NARROW and (dtype != "bf16" or pair):
        pytest.skip("the narrow tiles are bf16 single-CTA kernels")
    for K, kmajor in ((4096, True), (16384, True), (4096, False)):
        if bn not in T.plan_widths(dtype, pair, kmajor):
            continue
        monkeypatch.setenv("GB300_GEMM_BN", str(bn))
        monkeypatch.setenv("GB300_GEMM_PAIR", "1" if pair else "0")
        monkeypatch.setenv("GB300_GEMM_SPLITS", "1")
        G.gemm_reload_overrides()
        st, plan = G.gemm_plan_query(2048, 2048, K, dtype == "int8", 1 if kmajor else 0)
        assert st == 0 and plan["bn"] == bn
        kb_per = -(-K // 64)
        if dtype == "bf16":
            tma = 2 if bn == 224 else 1
            ew = 4
        else:
            tma = 1 if (bn not in (192, 224) or kb_per <= 128) else 0
            ew = 4 if bn == 128 else 8
        v = T.Variant(dtype, pair, bn, False, ew, tma)
        assert plan["stages"] == v.max_stages(), (v, plan)


def _shapes(n=300, seed=3):
    rng = random.Random(seed)
    out = []
    for _ in range(n):
        M = rng.choice([rng.randint(9, 300), rng.randint(300, 9000), 128 * rng.randint(1, 64)])
        N = rng.choice([rng.randint(16, 300), rng.randint(300, 13000), 64 * rng.randint(1, 160)])
        K = rng.choice([rng.randint(16, 1000), rng.randint(1000, 20000), 256 * rng.randint(1, 40)])
        out.append((M, N, K, rng.choice(["int8", "bf16"]), rng.choice([0, 1])))
    return out


def test_library_planner_equals_the_model(lib):
    """On 300 random shapes routed to the tensor-core kernels the library's
    choice of family, width and split is the model's (same candidates, same
    cost table, same tie rule)."""
    table = T.load_table()
    checked = 0
    for (M, N, K, dtype, layout) in _shapes():
        st, plan = G.gemm_plan_query(M, N, K, dtype == "int8", layout)
        assert st == 0
        if plan["route"] not in (G.GEMM_ROUTE_TC_SINGLE, G.GEMM_ROUTE_TC_PAIR):
            continue
        want = T.choose_plan(M, N, K, dtype, layout == 1, table)
        got = (plan["route"] == G.GEMM_ROUTE_TC_PAIR, plan["bn"], plan["splits"], plan["tail_splits"])
        assert got == T.plan_key(want), (M, N, K, dtype, layout, plan, want)
        assert plan["model_us"] == pytest.approx(T.plan_cost_us(M, N, K, dtype, want, table), rel=1e-4)
        assert plan["dram_us"] == pytest.approx(T.mem_time_us(M, N, K, dtype, want), rel=1e-6)
        checked += 1
    assert checked > 150


def test_plan_query_routes(lib):
    st, p = G.gemm_plan_query(0, 10, 10, True, 0)
    assert st == 0 and p["route"] == G.GEMM_ROUTE_NONE
    st, p = G.gemm_plan_query(10, 10, 0, False, 0)
    assert st == 0 and p["route"] == G.GEMM_ROUTE_ZERO_FILL
    st, p = G.gemm_plan_query(1, 11008, 4096, True, 0)
    assert st == 0 and p["route"] == G.GEMM_ROUTE_SMALL_M
    st, p = G.gemm_plan_query(128, 11008, 4096, True, 1)
    assert st == 0 and p["route"] == G.GEMM_ROUTE_SMALL_OPERAND and p["bn"] == 128
    st, p = G.gemm_plan_query(16, 4096, 4096, True, 0)      # B stored K x N, read transposed
    assert st == 0 and p["route"] == G.GEMM_ROUTE_SMALL_OPERAND and p["bn"] == 64
    st, p = G.gemm_plan_query(8192, 8192, 8192, False, 0)
    assert st == 0 and p["route"] in (G.GEMM_ROUTE_TC_SINGLE, G.GEMM_ROUTE_TC_PAIR) and p["grid"] > 0
    assert G.gemm_plan_query(4, 4, 131072, True, 0)[0] == G.GEMM_ERR_UNSUPPORTED
    assert G.gemm_plan_query(-1, 4, 4, True, 0)[0] == G.GEMM_ERR_INVALID_ARG
    assert G.gemm_plan_query(4, 4, 4, True, 2)[0] == G.GEMM_ERR_INVALID_ARG


def test_plan_query_split_tail(lib, monkeypatch):
    """Split tails on the host-only plan query: chosen by the model for
    8192^3 (1024 CTA-pair tiles on 76 pairs: 13 full rounds and 36 tiles in
    halves), turned off by GB300_GEMM_TAIL_SPLITS=0, forced to another
    split count where one fits (T = 3 does not fit 36 pair tiles into 76
    pairs: a single-CTA width takes it), and absent where the tiles fill no
    second round."""
    st, p = G.gemm_plan_query(8192, 8192, 8192, False, 0)
    assert st == 0 and p["route"] == G.GEMM_ROUTE_TC_PAIR and (p["bn"], p["splits"], p["tail_splits"]) == (256, 1, 2)
    monkeypatch.setenv("GB300_GEMM_TAIL_SPLITS", "0")
    G.gemm_reload_overrides()
    st, p = G.gemm_plan_query(8192, 8192, 8192, False, 0)
    assert st == 0 and p["tail_splits"] == 0
    monkeypatch.setenv("GB300_GEMM_TAIL_SPLITS", "3")
    G.gemm_reload_overrides()
    st, p = G.gemm_plan_query(8192, 8192, 8192, True, 0)
    assert st == 0 and p["tail_splits"] == 3 and p["route"] == G.GEMM_ROUTE_TC_SINGLE and p["splits"] == 1
    st, p = G.gemm_plan_query(1024, 1024, 1024, True, 1)   # 64 tiles: no second round
    assert st == 0 and p["tail_splits"] == 0


def _measurements():
    with open(T.MEASUREMENTS) as f:
        return json.load(f)


def test_planner_table_is_generated_from_the_committed_measurements():
    """csrc/plan_table.h is exactly what tile_model.py writes for
    plan_measurements.json: the table is fitted, not hand-entered."""
    meas = _measurements()
    text = T.header_text(T.fit(meas), os.path.basename(T.MEASUREMENTS))
    with open(T.HEADER) as f:
        assert f.read() == text


def test_model_fits_the_measurements():
    """The fitted model (Eq. 9 with measured eff per variant, the split and
    staging terms) reproduces the measured plans' times, and its choice is
    on average within 3 % of the best forced plan of each shape, never more
    than 25 % off."""
    meas = _measurements()
    table = T.fit(meas)
    assert table["fit"]["median_abs_rel_err"] < 0.08
    rep = T.evaluate(meas, table)
    ratios = np.array([r["model_us"] / r["best_us"] for r in rep])
    assert np.exp(np.mean(np.log(ratios))) < 1.03
    assert ratios.max() < 1.25
    eff = T.efficiency(table)
    assert all(0.2 < e < 1.05 for e in eff.values()), eff


def test_balanced_search_on_the_measurements():
    """The paper's iterative search (the model proposes the next plan, one
    measurement per step, stop at the first slowdown) reaches, on the
    measured plans, a plan within 5 % of the best for most shapes and within
    10 % for nearly all, after a few measurements."""
    meas = _measurements()
    table = T.fit(meas)
    close, steps = 0, []
    for s in meas["shapes"]:
        by = {T.plan_key(p): p["us"] for p in s["plans"]}
        best = min(by.values())
        plan, t, n = T.balanced_search(s["M"], s["N"], s["K"], s["dtype"], s["layout"] == "col",
                                       lambda p: by.get(T.plan_key(p), float("inf")), table,
                                       meas.get("sms"))
        steps.append(n)
        close += t <= 1.05 * best
        assert t <= 1.25 * best, s
    assert close >= 0.85 * len(meas["shapes"])
    assert np.median(steps) <= 4

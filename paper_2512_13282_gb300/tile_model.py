"""Tile-size model and balanced-point search of the paper (Sec. 4.5), restated
for one GB300, and the generator of the library's planner table.

The paper chooses its NPU kernel in two steps.  Per core (Sec. 4.5.1) it
bounds the tile m_ct x k_ct x n_ct by compute against DMA time (Eq. 1-4) and
by the L1 capacity (Eq. 5), and ranks the feasible tiles by MACs per tile,
then by the smallest output tile.  For the whole array (Sec. 4.5.2) it
models DRAM traffic (Eq. 6-8), compute and memory time (Eq. 9-10), and walks
from a memory-bound start towards the balanced point T_comp ~ T_mem,
measuring each step on the device and stopping at the first slowdown.

On GB300 the "core" is one SM running one persistent CTA (or two SMs running
a CTA pair on one 256-row tile); the tile is BM x BN per CTA, BK deep per
pipeline stage, accumulating in TMEM.  The restatement:

  Eq. 1  C_comp = BM_cta * BK * BN / (eff * MACS_PER_CLK)      cycles per stage
  Eq. 2  CA_comm = BM_cta * BK * ty(A) / TMA_BYTES_PER_CLK
  Eq. 3  CB_comm = BK * BN_cta * ty(B) / TMA_BYTES_PER_CLK
  Eq. 4  C_comp >= CA_comm + CB_comm   (one TMA engine per SM fills both
         operands, so the sum -- the paper's A and B DMA channels are separate)
  Eq. 5  STAGES * (BM_cta*BK*ty(A) + BK*BN_cta*ty(B)) + epilogue staging
         + barriers <= 227 KB of shared memory, and 2 * BN fp32 accumulator
         columns <= 512 TMEM columns (C lives in TMEM, double-buffered, not in
         the operand memory as on the NPU).  STAGES >= 2 (the paper's double
         buffer) and as many as fit: the library's stage counts are this
         maximum (max_stages).
  BK: one 128-byte swizzle row of bf16 (BK * ty = 128 B, the widest K extent
      of a swizzled TMA box row); a deeper K per stage is more stages.
  Eq. 6-8 A_mem = M*K*ty(A) * rA, B_mem = K*N*ty(B) * rB, C_mem = M*N*ty(C)
         (+ split-K partials written and read once), where the reuse factors
         rA, rB are 1 when the operands stay in the 129 MB L2 while the tiles
         that share them run (the grouped raster keeps 8 row tiles of A in
         L2 while it sweeps N; B is re-read once per group of row tiles when
         it does not fit), i.e. the paper's M*K*N/(n_ct*n_cols) with the
         reuse supplied by L2 instead of broadcast streams.
  Eq. 9  T_comp = rounds * (kb_per_unit * t_kstep + t_unit): the kernel runs
         ceil(tiles * S / slots) rounds of one unit (tile, K split) per slot;
         t_kstep = BK * BN * BM_cta / (eff * MACS_PER_CLK * clock), with eff
         measured per kernel variant, as the paper estimates eff from each
         previous measurement; t_unit is the per-unit start and epilogue.
  Eq. 10 T_mem = (A_mem + B_mem + C_mem) / DRAM_BW.
  Split-K, which the paper never uses, adds the partials' traffic and a
  reduction launch: T_split = r0 + r1 * (4 * S * M * N bytes).

With the 129 MB L2 supplying the reuse, T_mem hardly depends on the tile
(unlike the NPU's, where m_ct and n_ct set the DRAM traffic directly): it
classifies a GEMM (compute- or memory-bound, the paper's balance), and
separates plans only where B does not stay in L2 beside A and C and is
re-read once per group of row tiles (half as often with CTA pairs).  The
planner (csrc/gemm_api.cu make_plan) minimises T_comp + T_split + w * T_mem
over (family, BN, S) with the per-variant t_kstep and t_unit, the split
constants and the weight w of the DRAM time that the kernels do not hide,
which fit() derives from measurements (tile_sweep.py) and header_text()
writes to csrc/plan_table.h.  balanced_search() is the paper's
iterative procedure on the same candidates: the model proposes, measurements
decide, and the walk stops at the first slowdown.

    python -m paper_2512_13282_gb300.tile_model MEASUREMENTS.json   # fit, report, regenerate the header
"""
from __future__ import annotations

import json
import math
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
HEADER = os.path.join(HERE, "csrc", "plan_table.h")
MEASUREMENTS = os.path.join(HERE, "plan_measurements.json")

# GB300 resources (one GPU): SMs, co-resident SM pairs for one CTA per SM,
# dynamic shared memory per CTA, TMEM columns per SM, bf16 dense MACs per
# clock per SM (2.25 PFLOP/s nominal), L2->SM TMA fill per SM per clock
# (nominal), L2 capacity, maximum SM clock.
GB300 = {"sms": 152, "pair_slots": 76, "smem_per_cta": 232448, "tmem_cols": 512, "macs_per_clk": 4096,
         "tma_bytes_per_clk": 128, "l2_bytes": 129e6, "clock_ghz": 2.07, "hbm_gbs": 6693.8}

BM = 128          # rows of C per CTA (MMA M)
BK = 64           # K per pipeline stage: one 128-byte swizzle row of bf16
KB_DEPTH = BK
WIDTHS = (64, 96, 128, 192, 224, 256)
# the bf16 single-CTA kernels also come 64 and 96 wide (96 for B column-major
# only): tiles for memory-bound GEMMs with few rows, which fill the SMs
# without a K split; they do not meet Eq. 4 and are chosen only by time
NARROW = (64, 96)


class Variant:
    """One compiled tensor-core kernel: operand type of the epilogue, family
    (one CTA per 128-row tile, or a CTA pair per 256-row tile), tile width,
    epilogue warps and output staging (0: direct stores, 1: 4 KB TMA blocks
    per epilogue warp, 2: 1 KB blocks)."""

    def __init__(self, dtype, pair, bn, kmajor_only, epi_warps, tma_out):
        self.dtype, self.pair, self.bn = dtype, pair, bn
        self.kmajor_only, self.epi_warps, self.tma_out = kmajor_only, epi_warps, tma_out

    @property
    def bn_cta(self):
        return self.bn // 2 if self.pair else self.bn

    def stage_bytes(self):
        return BM * BK * 2 + self.bn_cta * BK * 2           # bf16 operands in shared memory

    def smem_bytes(self, stages):
        """Eq. 5: the operand ring, the epilogue's staging blocks, the
        barriers (2 per stage + 5) and the 1 KB alignment slack, as the
        kernels lay them out."""
        epi = {0: 0, 1: 4096, 2: 1024}[self.tma_out] * self.epi_warps
        return stages * self.stage_bytes() + epi + (2 * stages + 5) * 8 + 16 + 1024

    def max_stages(self):
        s = 1
        while self.smem_bytes(s + 1) <= GB300["smem_per_cta"]:
            s += 1
        return s

    def tmem_cols(self):
        c = 32
        while c < 2 * self.bn:
            c *= 2
        return c

    def eq4_cycles(self):
        """(C_comp at eff = 1, CA_comm + CB_comm) per stage, in SM cycles."""
        comp = BM * BK * self.bn / GB300["macs_per_clk"]
        comm = (BM * BK * 2 + BK * self.bn_cta * 2) / GB300["tma_bytes_per_clk"]
        return comp, comm

    def key(self):
        return (self.dtype, self.pair, self.bn, self.tma_out)

    def __repr__(self):
        return (f"{self.dtype} {'pair' if self.pair else 'single'} BN={self.bn} "
                f"{'direct' if self.tma_out == 0 else 'TMA'} stages={self.max_stages()}")


def compiled_variants():
    """The kernels the library instantiates (csrc/gemm_tc_*.cu,
    gemm_tc2_*.cu): bf16 with one epilogue warpgroup; int8 with two for
    tiles wider than 128; 224 (and the pair's 192) for B column-major only;
    the bf16 224-wide kernels stage through 1 KB blocks; the int8 192/224
    ones come with TMA staging blocks or with direct stores; and the narrow
    bf16 single-CTA tiles, 64 (both layouts) and 96 (B column-major)."""
    v = [Variant("bf16", False, 64, False, 4, 1), Variant("bf16", False, 96, True, 4, 1)]
    for pair in (False, True):
        for bn in WIDTHS:
            if bn in NARROW:
                continue
            km_only = bn == 224 or (pair and bn == 192)
            v.append(Variant("bf16", pair, bn, km_only, 4, 2 if bn == 224 else 1))
            ew = 4 if bn == 128 else 8
            v.append(Variant("int8", pair, bn, km_only, ew, 1))
            if bn in (192, 224):
                v.append(Variant("int8", pair, bn, km_only, ew, 0))
    return v


def single_core_ip(pair=False, dtype_bytes=2):
    """Sec. 4.5.1 on one SM: every (BM, BN, BK) the MMA and the swizzle
    allow that satisfies Eq. 4 and Eq. 5 with at least two stages, ranked by
    MACs per stage (descending), then by the output tile BM * BN
    (ascending)."""
    out = []
    for bm in ((128,) if not pair else (256,)):
        for bn in range(32, 257, 16):
            for bk in (16, 32, 64):
                if bk * dtype_bytes > 128:
                    continue
                bm_cta = bm // 2 if pair else bm
                bn_cta = bn // 2 if pair else bn
                stage = bm_cta * bk * dtype_bytes + bk * bn_cta * dtype_bytes
                if 2 * stage + 1024 > GB300["smem_per_cta"] or 2 * bn > GB300["tmem_cols"]:
                    continue
                comp = bm_cta * bk * bn / GB300["macs_per_clk"]
                comm = stage / GB300["tma_bytes_per_clk"]
                if comp < comm:
                    continue
                out.append({"bm": bm, "bn": bn, "bk": bk, "macs": bm * bn * bk, "c_tile": bm * bn,
                            "comp_cycles": comp, "comm_cycles": comm})
    out.sort(key=lambda r: (-r["macs"], r["c_tile"]))
    return out


def _ceil(a, b):
    return -(-a // b)


def plan_widths(dtype, pair, b_kmajor):
    """Tile widths compiled for one operand type, family and B layout, in
    the planner's order (widest first)."""
    if pair:
        return (256, 224, 192, 128) if b_kmajor else (256, 128)
    if b_kmajor:
        return (256, 224, 192, 128, 96, 64) if dtype == "bf16" else (256, 224, 192, 128)
    return (256, 192, 128, 64) if dtype == "bf16" else (256, 192, 128)


def candidate_plans(M, N, K, dtype, b_kmajor, sms=None, pair_slots=None):
    """Every (family, BN, S, tail split) the planner considers for an
    M x N x K GEMM, with its tile count, K steps per unit and rounds.  Pairs
    need M > 128; tiles wider than 128 only where N > 128; S keeps >= 4 K
    steps per unit and at most 2 units per slot.  After the splits of each
    width come its split-tail plans: whole tiles for the full rounds, the
    tiles of a last, partly filled round split in T = 2 .. 8 (tail x T at
    most one round, >= 4 K steps a unit)."""
    sms = sms or GB300["sms"]
    pair_slots = pair_slots if pair_slots is not None else GB300["pair_slots"]
    num_kb = _ceil(K, BK)
    out = []
    for pair in (False, True):
        if pair and (M <= BM or pair_slots <= 0):
            continue
        slots = pair_slots if pair else sms
        tiles_m = _ceil(M, 2 * BM if pair else BM)
        for bn in plan_widths(dtype, pair, b_kmajor):
            if N <= 128 and bn > 128:
                continue
            tiles = tiles_m * _ceil(N, bn)
            seen = set()
            for s in range(1, 17):
                kb_per = _ceil(num_kb, min(s, num_kb))
                s2 = _ceil(num_kb, kb_per)
                if s2 in seen:
                    continue
                if s2 > 1 and (kb_per < 4 or tiles * s2 > 2 * slots):
                    continue
                seen.add(s2)
                out.append({"pair": pair, "bn": bn, "splits": s2, "kb_per": kb_per, "tiles": tiles,
                            "rounds": _ceil(tiles * s2, slots), "tail_splits": 0})
            full, tail = divmod(tiles, slots)
            if full < 1 or tail == 0:
                continue
            for t in range(2, 9):
                if tail * t > slots:
                    break
                kb_tail = _ceil(num_kb, t)
                if _ceil(num_kb, kb_tail) != t or kb_tail < 4:
                    continue
                out.append({"pair": pair, "bn": bn, "splits": 1, "kb_per": num_kb, "tiles": tiles,
                            "rounds": full + 1, "tail_splits": t, "kb_tail": kb_tail, "tail": tail})
    return out


def plan_terms(M, N, plan):
    """(K steps, units) of the busiest CTA and MB of split-K partials of a
    plan: rounds x kb_per steps with split-K; the full rounds' steps plus one
    tail unit's with a split tail, whose partials cover only the tail tiles."""
    if plan.get("tail_splits", 0):
        rows = 2 * BM if plan["pair"] else BM
        steps = (plan["rounds"] - 1) * plan["kb_per"] + plan["kb_tail"]
        return steps, plan["rounds"], 4 * plan["tail_splits"] * plan["tail"] * rows * plan["bn"] / 1e6
    mb = 4 * plan["splits"] * M * N / 1e6 if plan["splits"] > 1 else 0.0
    return plan["rounds"] * plan["kb_per"], plan["rounds"], mb


def plan_key(plan):
    return (plan["pair"], plan["bn"], plan["splits"], plan.get("tail_splits", 0))


# ------------------------------------------------------------------ cost

def mem_time_us(M, N, K, dtype, plan):
    """Eq. 6-8 and 10 for one plan, in microseconds: A once (the grouped
    raster keeps a group's 8 row tiles of A in L2 while it sweeps N), B once
    if it fits in half the L2 or A, B and C together fit in L2 (C passes
    through L2 as the tiles store it), else once per group of 8 row tiles
    (128 or 256 rows each: CTA pairs halve the re-reads), C once.  Split-K
    partials are left out: they stay in L2, and their cost is the fitted
    split term."""
    ty = 2  # operands are bf16 in the kernel (int8 is staged as bf16)
    tyc = 4 if dtype == "int8" else 2
    l2 = GB300["l2_bytes"]
    a_bytes, b_bytes, c_bytes = M * K * ty, K * N * ty, M * N * tyc
    rows_per_group = 8 * (2 * BM if plan["pair"] else BM)
    fits = b_bytes <= l2 / 2 or a_bytes + b_bytes + c_bytes <= l2
    rb = 1.0 if fits else max(1.0, float(_ceil(M, rows_per_group)))
    return (a_bytes + b_bytes * rb + c_bytes) / (GB300["hbm_gbs"] * 1e3)


def plan_cost_us(M, N, K, dtype, plan, table):
    """T_comp + T_split (Eq. 9 with wave quantisation, and the split term)
    with the fitted per-variant costs of `table`: the time the planner
    minimises.  Eq. 10's DRAM time (mem_time_us) is reported beside it; with
    a 129 MB L2 it barely depends on the plan, so it does not rank plans."""
    g = table["groups"].get(group_key(dtype, plan["pair"], plan["bn"]))
    if g is None:
        return math.inf
    steps, rounds, mb = plan_terms(M, N, plan)
    t_comp = steps * g["kstep_us"] + rounds * g["unit_us"]
    t_split = 0.0
    if mb > 0:
        sp = table["split"][dtype]
        t_split = sp["fixed_us"] + sp["us_per_mb"] * mb
    return t_comp + t_split


def group_key(dtype, pair, bn):
    return f"{dtype}/{'pair' if pair else 'single'}/{bn}"


def rank_us(M, N, K, dtype, plan, table):
    """What the planner minimises: T_comp + T_split plus the share
    `mem_weight` of Eq. 10's DRAM time that the kernels do not hide -- which
    separates plans only where B is re-read (B does not stay in L2 beside A
    and C, and a CTA pair's 256-row groups re-read it half as often)."""
    return plan_cost_us(M, N, K, dtype, plan, table) + table.get("mem_weight", 0.0) * mem_time_us(M, N, K, dtype, plan)


def choose_plan(M, N, K, dtype, b_kmajor, table, sms=None, pair_slots=None):
    """The planner: the candidate of least rank_us (the first one, in
    candidate order, on a tie)."""
    best, best_c = None, math.inf
    for p in candidate_plans(M, N, K, dtype, b_kmajor, sms, pair_slots):
        c = rank_us(M, N, K, dtype, p, table)
        if c < best_c - 1e-9:
            best, best_c = p, c
    return best


# ------------------------------------------------------------------- fit

def staging_mb(M, N, K, dtype):
    """MB the int8 operand staging pass moves (1 byte read, 2 written per
    element of A and B); none for bf16."""
    return 3 * (M * K + K * N) / 1e6 if dtype == "int8" else 0.0


def fit(meas):
    """Least-squares fit of the per-variant K-step and unit costs, a launch
    constant per operand type, the int8 staging pass per MB and the split
    constants to the sweep:
        t = c0[dtype] + c1 * MB_staged + rounds * (kb_per * kstep_g + unit_g)
            + [S > 1] (r0[dtype] + r1[dtype] * MB_partials),
    each shape's plans weighted by 1 / sqrt(its best time): between relative
    errors (every shape alike) and absolute ones (the large GEMMs, which
    dominate any workload's time), the weighting whose choices come closest
    to the best forced plans of the sweep."""
    rows, rhs, weights = [], [], []
    shapes = meas["shapes"]
    groups = sorted({group_key(s["dtype"], p["pair"], p["bn"]) for s in shapes for p in s["plans"]})
    gidx = {g: i for i, g in enumerate(groups)}
    ng = len(groups)
    base = 3                      # c0 bf16, c0 int8, c1 (int8 staging per MB)
    ncol = base + 2 * ng + 4
    for s in shapes:
        best = min(p["us"] for p in s["plans"])
        d = 0 if s["dtype"] == "bf16" else 1
        for p in s["plans"]:
            r = np.zeros(ncol)
            r[d] = 1.0
            r[2] = staging_mb(s["M"], s["N"], s["K"], s["dtype"])
            gi = gidx[group_key(s["dtype"], p["pair"], p["bn"])]
            steps, rounds, mb = plan_terms(s["M"], s["N"], p)
            r[base + 2 * gi] = steps
            r[base + 2 * gi + 1] = rounds
            if mb > 0:
                r[base + 2 * ng + 2 * d] = 1.0
                r[base + 2 * ng + 2 * d + 1] = mb
            rows.append(r)
            rhs.append(p["us"])
            weights.append(1.0 / math.sqrt(best))
    A = np.array(rows) * np.array(weights)[:, None]
    b = np.array(rhs) * np.array(weights)
    x, *_ = np.linalg.lstsq(A, b, rcond=None)
    table = {"groups": {}, "split": {}, "launch_us": {"bf16": float(x[0]), "int8": float(x[1])},
             "staging_us_per_mb": float(x[2])}
    for g, i in gidx.items():
        table["groups"][g] = {"kstep_us": float(max(x[base + 2 * i], 1e-4)),
                              "unit_us": float(max(x[base + 2 * i + 1], 0.0))}
    for d, name in ((0, "bf16"), (1, "int8")):
        table["split"][name] = {"fixed_us": float(max(x[base + 2 * ng + 2 * d], 0.0)),
                                "us_per_mb": float(max(x[base + 2 * ng + 2 * d + 1], 0.0))}
    # The weight of the DRAM time in the ranking: the grid value in the
    # middle of the run of values whose choices take the least measured time
    # over the sweep (the choices change only at a few thresholds).
    totals = []
    for w in MEM_WEIGHTS:
        table["mem_weight"] = w
        totals.append(sum(r["model_us"] if r["model_us"] is not None else math.inf for r in evaluate(meas, table)))
    least = min(totals)
    run = [i for i, t in enumerate(totals) if t <= least + 1e-6]
    table["mem_weight"] = MEM_WEIGHTS[run[len(run) // 2]]
    pred = np.array(rows) @ x
    rel = (pred - np.array(rhs)) / np.array(rhs)
    table["fit"] = {"plans": len(rhs), "shapes": len(shapes), "rms_rel_err": float(np.sqrt(np.mean(rel ** 2))),
                    "median_abs_rel_err": float(np.median(np.abs(rel))),
                    "max_abs_rel_err": float(np.max(np.abs(rel)))}
    return table


MEM_WEIGHTS = (0.0, 0.025, 0.05, 0.1, 0.2, 0.4)


def predict_us(M, N, K, dtype, plan, table):
    """Modelled time of the whole GEMM (launch and int8 staging included)."""
    return (table["launch_us"][dtype] + table["staging_us_per_mb"] * staging_mb(M, N, K, dtype)
            + plan_cost_us(M, N, K, dtype, plan, table))


def efficiency(table):
    """eff of Eq. 1 per variant: the K step's MMA time at the nominal peak
    and maximum clock over the fitted K-step time."""
    out = {}
    for g, c in table["groups"].items():
        dtype, fam, bn = g.split("/")
        macs = BM * BK * int(bn) * (2 if fam == "pair" else 1)
        slots_per_unit = 2 if fam == "pair" else 1
        ideal_us = macs / (GB300["macs_per_clk"] * slots_per_unit) / (GB300["clock_ghz"] * 1e3)
        out[g] = ideal_us / c["kstep_us"]
    return out


def evaluate(meas, table):
    """Per shape: the measured time of the model's choice, of the planner
    built into the library at measurement time, and of the best forced plan."""
    rep = []
    for s in meas["shapes"]:
        choice = choose_plan(s["M"], s["N"], s["K"], s["dtype"], s["layout"] == "col", table, meas.get("sms"))
        by = {plan_key(p): p["us"] for p in s["plans"]}
        best = min(s["plans"], key=lambda p: p["us"])
        rep.append({"shape": f"{s['dtype']} {s['M']}x{s['N']}x{s['K']} {s['layout']}",
                    "model_us": by.get(plan_key(choice)),
                    "planner_us": s["planner_us"], "best_us": best["us"],
                    "model_choice": plan_key(choice), "best": plan_key(best)})
    return rep


def balanced_search(M, N, K, dtype, b_kmajor, measure, table, sms=None, pair_slots=None):
    """The paper's iterative search (Sec. 4.5.2) on GB300's knobs.  The paper
    proposes each step's configuration from its model (an IP solved for the
    next k_ct), measures it on the device, and stops as soon as a step is
    slower than the one before.  Here the model ranks every candidate (family,
    BN, S) by modelled time; the steps measure them in that order --
    `measure(plan)` returns the measured time -- until the first measured
    slowdown.  Returns (best plan measured, its time, plans measured)."""
    cands = candidate_plans(M, N, K, dtype, b_kmajor, sms, pair_slots)
    cands.sort(key=lambda q: plan_cost_us(M, N, K, dtype, q, table))
    best, best_t, prev, n = None, math.inf, math.inf, 0
    for p in cands:
        t = measure(p)
        n += 1
        if t < best_t:
            best, best_t = p, t
        if n > 1 and t > prev:
            break
        prev = t
    return best, best_t, n


# --------------------------------------------------------------- header

def header_text(table, source="plan_measurements.json"):
    lines = [
        "// plan_table.h -- GENERATED by paper_2512_13282_gb300/tile_model.py from",
        f"// {source} (tile_sweep.py on one GB300); do not edit by hand.",
        "//",
        "// Per compiled tensor-core kernel variant: the fitted time of one K step of",
        "// BK = 64 (eff of Eq. 1 measured) and the fixed time of one unit (start and",
        "// epilogue), in microseconds; and per operand type the split-K terms",
        "// (reduction launch, and time per MB of fp32/int32 partials).  The planner",
        "// minimises the busiest CTA's K steps * kstep + its units * unit + split",
        "// terms (Eq. 9 with wave quantisation; a split tail adds one round of a",
        "// tail unit's steps to the full rounds) + kMemWeight * the DRAM time of",
        "// Eq. 6-8, 10 (the share of B's re-reads the kernels do not hide).",
        "#pragma once",
        "",
        "namespace gb300 {",
        "namespace plan_table {",
        "",
        "struct StepCost {",
        "  float kstep_us;  // one K step of 64 for one unit",
        "  float unit_us;   // per unit: start, accumulator drain, stores",
        "};",
        "",
        "// [0 bf16, 1 int8][0 single CTA, 1 CTA pair][BN %s]; {0, 0}: not compiled" % ", ".join(map(str, WIDTHS)),
        "constexpr StepCost kCost[2][2][%d] = {" % len(WIDTHS),
    ]
    for dtype in ("bf16", "int8"):
        lines.append("    {")
        for fam in ("single", "pair"):
            cells = []
            for bn in WIDTHS:
                g = table["groups"].get(f"{dtype}/{fam}/{bn}")
                cells.append("{%.5ff, %.4ff}" % (g["kstep_us"], g["unit_us"]) if g else "{0.0f, 0.0f}")
            lines.append("        {" + ", ".join(cells) + "},")
        lines.append("    },")
    lines += [
        "};",
        "",
        "// split-K: [0 bf16, 1 int8]",
        "constexpr float kSplitFixedUs[2] = {%.4ff, %.4ff};" % (table["split"]["bf16"]["fixed_us"],
                                                               table["split"]["int8"]["fixed_us"]),
        "constexpr float kSplitUsPerMB[2] = {%.5ff, %.5ff};" % (table["split"]["bf16"]["us_per_mb"],
                                                               table["split"]["int8"]["us_per_mb"]),
        "",
        "// Eq. 10: DRAM bandwidth (GB/s) and the L2 capacity the reuse factors use.",
        "constexpr double kHbmGBs = %.1f;" % GB300["hbm_gbs"],
        "constexpr double kL2Bytes = %.1f;" % GB300["l2_bytes"],
        "constexpr double kMemWeight = %.3f;" % table["mem_weight"],
        "",
        "}  // namespace plan_table",
        "}  // namespace gb300",
        "",
    ]
    return "\n".join(lines)


def table_from_header(text):
    """Parse the generated header back (tests compare it with a fresh fit)."""
    import re
    nums = [float(x) for x in re.findall(r"([0-9.]+)f", text.split("kCost")[1].split("};")[0])]
    table = {"groups": {}, "split": {}}
    i = 0
    for dtype in ("bf16", "int8"):
        for fam in ("single", "pair"):
            for bn in WIDTHS:
                k, u = nums[i], nums[i + 1]
                i += 2
                if k > 0:
                    table["groups"][f"{dtype}/{fam}/{bn}"] = {"kstep_us": k, "unit_us": u}
    fx = [float(x) for x in re.findall(r"kSplitFixedUs\[2\] = \{([0-9.]+)f, ([0-9.]+)f\}", text)[0]]
    pm = [float(x) for x in re.findall(r"kSplitUsPerMB\[2\] = \{([0-9.]+)f, ([0-9.]+)f\}", text)[0]]
    table["split"] = {"bf16": {"fixed_us": fx[0], "us_per_mb": pm[0]}, "int8": {"fixed_us": fx[1], "us_per_mb": pm[1]}}
    table["mem_weight"] = float(re.findall(r"kMemWeight = ([0-9.]+);", text)[0])
    return table


def load_table():
    """The table compiled into the library (parsed from the header)."""
    with open(HEADER) as f:
        return table_from_header(f.read())


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
    path = argv[0] if argv else MEASUREMENTS
    with open(path) as f:
        meas = json.load(f)
    table = fit(meas)
    with open(HEADER, "w") as f:
        f.write(header_text(table, os.path.basename(path)))
    rep = evaluate(meas, table)
    ratios = [r["model_us"] / r["best_us"] for r in rep if r["model_us"]]
    old = [r["planner_us"] / r["best_us"] for r in rep]
    print(json.dumps({"fit": table["fit"], "split": table["split"],
                      "eff": {k: round(v, 3) for k, v in efficiency(table).items()},
                      "model_choice_over_best_geomean": float(np.exp(np.mean(np.log(ratios)))),
                      "model_choice_over_best_max": float(max(ratios)),
                      "planner_at_measurement_over_best_geomean": float(np.exp(np.mean(np.log(old))))}, indent=1))


if __name__ == "__main__":
    main()

"""Measure every forced tile plan of the tensor-core GEMM kernels on one GPU.

This is the measurement half of the balanced-point search (Sec. 4.5: the
starting values and each step's efficiency are measured on the device).  For
each shape of a fixed set -- the tensor-core GEMMs of the benchmark
workloads and a seeded sample of the roofline sweep sizes -- every plan the
library can be forced into (kernel family: one CTA per 128-row tile or a CTA
pair per 256-row tile; tile width BN; split-K factor S; split tail T) is timed with CUDA
events after a 512 MiB L2 flush: the mean of `reps` launches without the
fastest and the slowest (the event clock advances in steps of about 1 us on
GB300, so a median of a few launches of a 10-30 us GEMM is off by up to a
step; a mean of many is not).  The result is written as JSON; tile_model.py
fits the planner's cost table to it.

    python -m paper_2512_13282_gb300.tile_sweep OUT.json [--reps 15] [--sample 40]

Needs a GPU and the built library.  Results of int8 GEMMs are exact whatever
the plan, and bf16 results differ only in summation order, so no plan is
checked here; the GPU tests cover every family, width and split.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import sys
import time

import numpy as np

from . import workloads as W
from .tile_model import candidate_plans, GB300

ENV_KEYS = ("GB300_GEMM_BN", "GB300_GEMM_PAIR", "GB300_GEMM_SPLITS", "GB300_GEMM_TAIL_SPLITS",
            "GB300_GEMM_SKINNY_MAX_M", "GB300_GEMM_S8TM", "GB300_GEMM_TINY_MAX_MACS")
# every int8 GEMM of the sweep on the tensor-core kernels
TC_ONLY = {"GB300_GEMM_SKINNY_MAX_M": 0, "GB300_GEMM_S8TM": 0, "GB300_GEMM_TINY_MAX_MACS": 0}


def sweep_shapes(sample: int = 40, seed: int = 11):
    """(M, N, K, dtype, layout) of the sweep: the workloads' GEMMs with M > 8
    that the tensor-core kernels run (int8-int32 and bf16), then `sample`
    roofline sizes (both dtypes, B column-major) drawn with `seed`."""
    seen, out = set(), []
    for wl in ("square_sweep_512_4096", "square_8192", "transformer_projections", "irregular_skinny",
               "int8_square_256"):
        for g in W.WORKLOADS[wl].gemms:
            if g.M <= 8 or g.dtype not in ("int8", "bf16"):
                continue
            key = (g.M, g.N, g.K, g.dtype, g.layout)
            if key not in seen:
                seen.add(key)
                out.append(key)
    rng = np.random.default_rng(seed)
    sizes = W.roofline_sweep_sizes()
    for i in rng.choice(len(sizes), sample, replace=False):
        M, N, K = sizes[int(i)]
        for dt in ("int8", "bf16"):
            key = (M, N, K, dt, W.B_COL_MAJOR)
            if key not in seen:
                seen.add(key)
                out.append(key)
    return out


def main(argv=None):
    import torch

    from . import build as Bld
    from . import gemm as G

    ap = argparse.ArgumentParser()
    ap.add_argument("out")
    ap.add_argument("--reps", type=int, default=15)
    ap.add_argument("--sample", type=int, default=40)
    args = ap.parse_args(argv)
    Bld.build()
    G.library()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    flush = torch.empty((512 << 20) // 4, dtype=torch.float32, device=dev)
    st = torch.cuda.current_stream()
    shapes = sweep_shapes(args.sample)
    big = max(max(m * k, k * n) for m, n, k, _, _ in shapes)
    dA = torch.from_numpy(W.random_int8((big,), 31)).to(dev)
    dB = torch.from_numpy(W.random_int8((big,), 32)).to(dev)
    hA16 = torch.from_numpy(W.random_bf16((big,), 33).view(np.int16)).to(dev)
    hB16 = torch.from_numpy(W.random_bf16((big,), 34).view(np.int16)).to(dev)
    dC = torch.empty(max(m * n for m, n, _, _, _ in shapes) * 4, dtype=torch.uint8, device=dev)

    def setenv(d):
        for k in ENV_KEYS:
            os.environ.pop(k, None)
        for k, v in d.items():
            os.environ[k] = str(v)
        G.gemm_reload_overrides()

    def time_plan(M, N, K, dtype, layout):
        ldb = N if layout == W.B_ROW_MAJOR else K
        if dtype == "int8":
            fn, A, B, C = G.gemm_s8s8_s32, dA, dB, dC.view(torch.int32)
        else:
            fn, A, B, C = G.gemm_bf16_f32acc_bf16, hA16, hB16, dC.view(torch.int16)
        ts = []
        for r in range(args.reps + 2):
            flush.fill_(float(r))
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(st)
            rc = fn(M, N, K, A, K, B, ldb, layout, C, N, st)
            b.record(st)
            if rc != 0:
                raise RuntimeError(f"{dtype} {M}x{N}x{K}: {G.gemm_status_string(rc)}")
            if r >= 2:
                ts.append((a, b))
        torch.cuda.synchronize()
        us = sorted(x.elapsed_time(y) * 1e3 for x, y in ts)
        return statistics.mean(us[1:-1]) if len(us) > 2 else statistics.mean(us)

    rows = []
    t0 = time.time()
    for (M, N, K, dtype, layout) in shapes:
        setenv(TC_ONLY)
        default_us = time_plan(M, N, K, dtype, layout)
        plans = []
        for c in candidate_plans(M, N, K, dtype, layout == W.B_COL_MAJOR, sms=sms, pair_slots=GB300["pair_slots"]):
            setenv(dict(TC_ONLY, GB300_GEMM_PAIR=int(c["pair"]), GB300_GEMM_BN=c["bn"],
                        GB300_GEMM_SPLITS=c["splits"], GB300_GEMM_TAIL_SPLITS=c["tail_splits"]))
            plans.append(dict(c, us=round(time_plan(M, N, K, dtype, layout), 3)))
        best = min(plans, key=lambda p: p["us"])
        print(f"{dtype:4s} {M}x{N}x{K} {'col' if layout else 'row'}: planner {default_us:8.1f} us, best forced "
              f"{best['us']:8.1f} ({'pair' if best['pair'] else 'single'} BN={best['bn']} S={best['splits']} "
              f"T={best['tail_splits']})",
              file=sys.stderr, flush=True)
        rows.append({"M": M, "N": N, "K": K, "dtype": dtype, "layout": "col" if layout else "row",
                     "planner_us": round(default_us, 3), "plans": plans})
    setenv({})
    with open(args.out, "w") as f:
        json.dump({"device": torch.cuda.get_device_name(dev), "sms": sms, "reps": args.reps,
                   "flush": "512 MiB write before every launch", "statistic": "mean without min and max",
                   "seconds": round(time.time() - t0, 1),
                   "shapes": rows}, f, indent=0)


if __name__ == "__main__":
    main()

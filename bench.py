"""Benchmark of the GB300 dense GEMM library (C = A.B, int8->int32 exact and
bf16->fp32->bf16 RNE).

One step = every GEMM of the chosen workload once (default: all 37 GEMMs of
the five benchmark configurations -- int8 256^3, the square sweep
512..4096 of both paths, 8192^3 of both paths, the transformer projections
and the irregular/skinny shapes).  Inputs are seeded synthetic matrices
(workloads.py) resident in HBM before timing.  L2 (129 MB) is flushed by
writing a 512 MiB buffer before every timed GEMM; each GEMM is bracketed by
CUDA events on its stream, so flushes are not timed.  The flush leaves dirty
lines in L2 whose write-back lands in the next GEMM, so a second pass times
every GEMM again after a clean flush (the same write, then a 256 MiB read of
another buffer) and reports both per GEMM.  For HBM-bound GEMMs, the time of
a plain read of the same compulsory bytes after the same flush (the
library's read-bandwidth diagnostic: 16-byte loads, nothing kept) is measured
beside it: the ceiling an isolated call of that size can reach.  HBM-bound
GEMMs are also timed back to back (`ms_stream`): R calls on R distinct copies
of the operands, R x the compulsory bytes >= 384 MB (inputs larger than L2,
no flush), between one pair of events -- the per-call time a loop of such
GEMMs sees once launches overlap.

  value       whole-job throughput, sum(2*M*N*K) / sum(event time), in TOPS
              (tera-ops/s; int8 MACs and bf16 FMAs both count 2 ops)
  e2e         the same through the C ABI from pinned HOST buffers: per step,
              H2D copies of every A and B, the GEMMs, D2H of every C, all
              inside the timed region; copies run on two copy streams and
              overlap the other GEMMs' kernels, and a GEMM with a large C is
              issued as row blocks (the same call on rows of A and C) so
              that its results start down while later rows compute
  roofline    the dominant kernel (largest share of step time): the main
              kernel of one GEMM (tensor-core, or CUDA-core for tiny M), timed
              through the library's profiling events in a second pass of the
              same K steps right after the timed ones, against the
              measured bf16 peak (tensor-bound) or HBM copy bandwidth
  cpu_baseline  the CPU oracle on a bounded sample (whole rows of C) of the
              same GEMMs, on this host's cores

``--impl reference`` times the CPU oracle itself (the only reference this
path has) on bounded samples of the same workload.

Multi-GPU (torchrun): every rank runs the same workload on its own GPU
(replicas; the GEMM has no exchange step), value = all ranks' ops / max time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2512_13282_gb300 import workloads as W  # noqa: E402

METRIC = "int8 TOPS & bf16 TFLOPS per GEMM shape, 1 GB300; % of dense tensor-core peak"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FLUSH_BYTES = 512 << 20
STREAM_BYTES = 384 << 20
CLEAN_READ_BYTES = 256 << 20


def load_peaks():
    try:
        with open(PEAKS_FILE) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return dict(FALLBACK), "fallback"


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons in the background."""
    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        self.lines += [l for l in out.splitlines() if l.strip()]

    def summary(self):
        rows = []
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 8:
                continue
            if self.uuid and f[0] != self.uuid and not self.uuid.endswith(f[0]) and not f[0].endswith(self.uuid):
                continue
            try:
                rows.append((float(f[1]), float(f[2]), f[4:8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i in range(4) if r[i].lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# -------------------------------------------------------------- our path

class GemmCase:
    def __init__(self, g: W.Gemm, dev):
        from paper_2512_13282_gb300 import gemm as G
        self.g, self.G = g, G
        A, B = W.make_inputs(g)
        if g.dtype == "int8":
            ha, hb = torch.from_numpy(A), torch.from_numpy(B)
            self.C = torch.empty((g.M, g.N), dtype=torch.int32, device=dev)
            self.fn = G.gemm_s8s8_s32
        elif g.int8_in:  # int8-int16 / int8-int8: requantised outputs
            ha, hb = torch.from_numpy(A), torch.from_numpy(B)
            s16 = g.dtype == "int8_int16"
            self.C = torch.empty((g.M, g.N), dtype=torch.int16 if s16 else torch.int8, device=dev)
            narrow = G.gemm_s8s8_s16 if s16 else G.gemm_s8s8_s8

            def fn(M, N, K, A_, lda, B_, ldb, layout, C_, ldc, stream):
                return narrow(M, N, K, A_, lda, B_, ldb, layout, C_, ldc, g.shift, stream)
            self.fn = fn
        else:
            ha, hb = torch.from_numpy(A.view(np.int16)), torch.from_numpy(B.view(np.int16))
            self.C = torch.empty((g.M, g.N), dtype=torch.int16, device=dev)
            self.fn = G.gemm_bf16_f32acc_bf16
        self.A, self.B = ha.to(dev), hb.to(dev)
        self.hA, self.hB = ha.pin_memory(), hb.pin_memory()
        self.hC = torch.empty(self.C.shape, dtype=self.C.dtype).pin_memory()
        self.ldb = g.N if g.layout == W.B_ROW_MAJOR else g.K
        self.h2d = self.hA.numel() * self.hA.element_size() + self.hB.numel() * self.hB.element_size()
        self.d2h = self.hC.numel() * self.hC.element_size()

    def launch(self, A=None, B=None, C=None):
        g = self.g
        st = self.fn(g.M, g.N, g.K, self.A if A is None else A, g.K, self.B if B is None else B, self.ldb,
                     g.layout, self.C if C is None else C, g.N, None)
        if st != 0:
            raise RuntimeError(f"{g.name}: {self.G.gemm_status_string(st)}")

    def row_blocks(self, min_bytes=128 << 20, block_bytes=16 << 20, max_blocks=8):
        """Row ranges [r0, r1) of A and C for the host-buffer pass.  A C of
        at least `min_bytes` (over 0.6 ms on the download link) goes in
        blocks of about `block_bytes` (at most `max_blocks`, multiples of 256
        rows), so that its first rows travel back while later rows are
        computed; smaller ones stay whole, since each block costs a launch
        and, for int8, staging B again (measured: blocking the 4096^3 GEMMs
        made the square sweep's host-buffer pass slower, the 8192^3 ones
        made theirs faster)."""
        M = self.g.M
        if self.d2h < min_bytes:
            return [(0, M)]
        k = max(1, min(max_blocks, self.d2h // block_bytes))
        rows = -(-M // k)
        rows = -(-rows // 256) * 256
        return [(r0, min(M, r0 + rows)) for r0 in range(0, M, rows)]

    def launch_rows(self, r0, r1):
        """The GEMM restricted to rows [r0, r1) of A and C (the same call on
        a sub-matrix: A and C advance by whole rows, B is shared)."""
        g = self.g
        pa = self.A.data_ptr() + r0 * g.K * self.A.element_size()
        pc = self.C.data_ptr() + r0 * g.N * self.C.element_size()
        st = self.fn(r1 - r0, g.N, g.K, pa, g.K, self.B, self.ldb, g.layout, pc, g.N, None)
        if st != 0:
            raise RuntimeError(f"{g.name} rows {r0}..{r1}: {self.G.gemm_status_string(st)}")

    def time_back_to_back(self, stream, min_bytes, reps=5):
        """(median ms per call, copies): R calls back to back on R distinct
        device copies of A, B and C with R x compulsory bytes >= min_bytes,
        so that each call finds its operands outside L2 without a flush
        between calls; checked against the single call's result."""
        g = self.g
        copies = int(max(3, min(64, -(-min_bytes // max(1, compulsory_bytes(g))))))
        As = [self.A.clone() for _ in range(copies)]
        Bs = [self.B.clone() for _ in range(copies)]
        Cs = [torch.empty_like(self.C) for _ in range(copies)]
        for r in range(copies):  # untimed: plans and workspace settle
            self.launch(As[r], Bs[r], Cs[r])
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for r in range(copies):
                self.launch(As[r], Bs[r], Cs[r])
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b) / copies)
        self.launch()
        torch.cuda.synchronize()
        if g.dtype == "bf16":
            x, y = Cs[-1].view(torch.bfloat16).float(), self.C.view(torch.bfloat16).float()
            same = bool(torch.all((x - y).abs() <= 2.0 ** -7 * torch.maximum(x.abs(), y.abs())))
        else:
            same = torch.equal(Cs[-1], self.C)
        if not same:
            raise RuntimeError(f"{g.name}: back-to-back result differs from the single call")
        del As, Bs, Cs
        return statistics.median(ts), copies

    def launch_e2e(self):
        self.A.copy_(self.hA, non_blocking=True)
        self.B.copy_(self.hB, non_blocking=True)
        self.launch()
        self.hC.copy_(self.C, non_blocking=True)


def run_ours(args, rank, world, dev):
    from paper_2512_13282_gb300 import build as Bld
    from paper_2512_13282_gb300 import gemm as G
    Bld.build()
    G.library()
    wl = select(args)
    cases = [GemmCase(g, dev) for g in wl.gemms]
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    clean = torch.ones(CLEAN_READ_BYTES // 4, dtype=torch.float32, device=dev)
    sink = torch.empty((), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def do_flush(i, clean_l2=False):
        flush.fill_(float(i))
        if clean_l2:  # read another buffer: the flush's dirty lines are written back now
            torch.sum(clean, dim=0, out=sink)

    def step(times=None, kern=None, clean_l2=False):
        for i, c in enumerate(cases):
            do_flush(i, clean_l2)
            if times is not None:
                s, e = times[i]
                s.record(stream)
            if kern is not None:
                G.gemm_profile_events(*kern[i])
            c.launch()
            if kern is not None:
                G.gemm_profile_events(None, None)
            if times is not None:
                e.record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in cases] for _ in range(args.steps)]
    kev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in cases] for _ in range(args.steps)]
    for row in kev:  # materialise the event handles
        for s, e in row:
            s.record(stream)
            e.record(stream)
    torch.cuda.synchronize()

    uuid = str(getattr(torch.cuda.get_device_properties(dev), "uuid", "") or "")
    if uuid and not uuid.startswith("GPU-"):
        uuid = "GPU-" + uuid
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    launches0 = G.gemm_launch_count()
    t0 = time.perf_counter()
    for k in range(args.steps):
        step(ev[k])
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    launches = G.gemm_launch_count() - launches0
    if world > 1:
        torch.distributed.barrier()
    # Kernel-duration pass: the same steps again, with events bracketing each
    # GEMM's main kernel.  Kept out of the timed steps because an event
    # recorded between the staging kernel and the GEMM would cut their
    # programmatic-launch overlap.
    for k in range(args.steps):
        step(None, kev[k])
    torch.cuda.synchronize()
    # Clean-flush pass: the same steps after a flush that leaves L2 clean.
    cev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in cases] for _ in range(args.steps)]
    for k in range(args.steps):
        step(cev[k], clean_l2=True)
    torch.cuda.synchronize()
    # Read ceiling of the HBM-bound GEMMs: a plain read of the same bytes
    # after the same (dirty) flush (outside the timed steps).
    peaks, peak_src = load_peaks()
    bf16_peak = float(peaks.get("bf16_tflops", FALLBACK["bf16_tflops"]))
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK["hbm_gbs"]))
    read_ms = {}
    for i, c in enumerate(cases):
        if bound_of(c.g, bf16_peak, hbm_peak) != "hbm":
            continue
        nbytes = compulsory_bytes(c.g) // 16 * 16
        buf = torch.ones(nbytes // 4, dtype=torch.float32, device=dev)
        evs = []
        for k in range(args.steps + 2):
            do_flush(i)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            G.check(G.gemm_selftest_read_stream(buf, nbytes, stream))
            b.record(stream)
            if k >= 2:
                evs.append((a, b))
        torch.cuda.synchronize()
        read_ms[i] = statistics.mean(x.elapsed_time(y) for x, y in evs)
        del buf
    # Back-to-back pass of the HBM-bound GEMMs (outside the timed steps):
    # R calls on R distinct operand copies whose bytes together exceed L2.
    stream_ms = {}
    if not args.no_stream:
        for i, c in enumerate(cases):
            if bound_of(c.g, bf16_peak, hbm_peak) == "hbm":
                stream_ms[i] = c.time_back_to_back(stream, STREAM_BYTES)
    # the timed region is short: keep sampling clocks over the same work for
    # about a second more so the clock record has samples under load
    t1 = time.perf_counter()
    while time.perf_counter() - t1 < 1.0:
        step()
    torch.cuda.synchronize()
    sampler.stop()

    per_gemm_ms = [[ev[k][i][0].elapsed_time(ev[k][i][1]) for k in range(args.steps)] for i in range(len(cases))]
    per_kern_ms = [[kev[k][i][0].elapsed_time(kev[k][i][1]) for k in range(args.steps)] for i in range(len(cases))]
    per_clean_ms = [[cev[k][i][0].elapsed_time(cev[k][i][1]) for k in range(args.steps)] for i in range(len(cases))]
    gemm_ms = sum(sum(x) for x in per_gemm_ms) / args.steps  # device ms per step
    ops = sum(c.g.flops for c in cases)

    # e2e: host buffers, copies inside the timed region.  Within a step the
    # inputs of every GEMM go up on one copy stream, each GEMM (the public
    # C-ABI call, on the current stream) starts when its own inputs have
    # landed, and each result comes back on a second copy stream as soon as
    # its GEMM is done -- transfers of one GEMM overlap the kernels of the
    # others, as a caller batching GEMMs would arrange it.
    e2e_ms = None
    if not args.no_e2e:
        h2d = torch.cuda.Stream(device=dev)
        d2h = torch.cuda.Stream(device=dev)
        # The host link, not the GPU, bounds this path, and uploads and
        # downloads can share it in both directions at once.  Small GEMMs go
        # first (short wait for the first inputs) and last (short wait for the
        # last result), the large ones in the middle, where one GEMM's result
        # travels down while the next GEMM's inputs travel up.
        by_size = sorted(cases, key=lambda c: c.h2d + c.d2h)
        e2e_cases = by_size[0::2] + by_size[1::2][::-1]

        # A GEMM whose C is large goes as row blocks (B once, then A rows,
        # the call on those rows, their C rows back): its first results
        # travel down while the later blocks still compute.  The views and
        # events are made once, so that a step only enqueues work.
        plan = []  # per GEMM: (case, B copy, [(A rows copy, C rows copy, r0, r1, uploaded, done)])
        for c in e2e_cases:
            bl = c.row_blocks()
            whole = len(bl) == 1
            items = [(c.A[r0:r1], c.hA[r0:r1], c.hC[r0:r1], c.C[r0:r1], None if whole else (r0, r1),
                      torch.cuda.Event(), torch.cuda.Event()) for (r0, r1) in bl]
            plan.append((c, items))

        def e2e_step(start, stop):
            start.record(stream)
            h2d.wait_stream(stream)
            with torch.cuda.stream(h2d):
                for c, items in plan:
                    c.B.copy_(c.hB, non_blocking=True)
                    for (da, ha, hc, dc, rows, up, done) in items:
                        da.copy_(ha, non_blocking=True)
                        up.record(h2d)
            for c, items in plan:
                for (da, ha, hc, dc, rows, up, done) in items:
                    stream.wait_event(up)
                    if rows is None:
                        c.launch()
                    else:
                        c.launch_rows(*rows)
                    done.record(stream)
            with torch.cuda.stream(d2h):
                for c, items in plan:
                    for (da, ha, hc, dc, rows, up, done) in items:
                        d2h.wait_event(done)
                        hc.copy_(dc, non_blocking=True)
            stream.wait_stream(d2h)
            stop.record(stream)

        for _ in range(2):
            e2e_step(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        torch.cuda.synchronize()
        e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(args.steps)]
        issue_s = []
        for k in range(args.steps):
            flush.fill_(float(k))
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            e2e_step(*e_ev[k])
            issue_s.append(time.perf_counter() - t0)
        torch.cuda.synchronize()
        e2e_ms = sum(a.elapsed_time(b) for a, b in e_ev) / args.steps
        if rank == 0:
            print(f"e2e: {e2e_ms:.3f} ms per step on the device clock, {1e3 * statistics.median(issue_s):.3f} ms "
                  "to issue a step on the host", file=sys.stderr)
        # The results that came back through the row blocks equal those of
        # one whole-matrix call (int8: bit for bit; bf16: the blocks may
        # split K differently, so each is within the accumulation bound of
        # the exact sum -- 2^-8 of it plus 2^-20 of the sum of |a b| -- and
        # they are within twice that of each other).
        for c in e2e_cases:
            c.launch()
            whole = c.C.cpu()
            got = c.hC.clone()
            if c.g.dtype == "bf16":
                a = whole.view(torch.bfloat16).float()
                b = got.view(torch.bfloat16).float()
                a_abs = c.A.view(torch.bfloat16).float().abs()
                b_abs = c.B.view(torch.bfloat16).float().abs()
                mag = (a_abs @ (b_abs if c.g.layout == W.B_ROW_MAJOR else b_abs.t())).cpu()
                del a_abs, b_abs
                ok = bool(torch.all((a - b).abs() <= 2.0 ** -7 * torch.maximum(a.abs(), b.abs()) + 2.0 ** -19 * mag))
            else:
                ok = torch.equal(whole, got)
            if not ok:
                raise RuntimeError(f"{c.g.name}: host-buffer results differ from the whole-matrix call")

    gemm_ms, e2e_max, wall = max_over_ranks([gemm_ms, e2e_ms or 0.0, wall], world, dev)

    # Means over the steps: event-timed GEMMs of a few tens of microseconds
    # right after the flush come out on a grid of about 2 us on GB300 (the
    # events themselves resolve 32 ns), so a median lands on a grid point;
    # the samples spread over neighbouring points, and their mean resolves
    # the time between them.
    per = []
    for i, c in enumerate(cases):
        ms = statistics.mean(per_gemm_ms[i])
        kms = statistics.mean(per_kern_ms[i])
        cms = statistics.mean(per_clean_ms[i])
        tops = c.g.flops / (ms * 1e-3) / 1e12
        gbps = compulsory_bytes(c.g) / (ms * 1e-3) / 1e9
        row = {"gemm": c.g.name, "bound": bound_of(c.g, bf16_peak, hbm_peak), "ms": round(ms, 5),
               "main_kernel_ms": round(kms, 5), "tops": round(tops, 2),
               "frac_of_bf16_peak": round(tops / bf16_peak, 4), "gbps": round(gbps, 1),
               "frac_of_hbm": round(gbps / hbm_peak, 4), "best_ms": round(min(per_gemm_ms[i]), 5),
               "ms_clean_l2": round(cms, 5),
               "frac_of_hbm_clean_l2": round(compulsory_bytes(c.g) / (cms * 1e-3) / 1e9 / hbm_peak, 4)}
        if i in stream_ms:
            t_stream, copies = stream_ms[i]
            row["ms_stream"] = round(t_stream, 5)
            row["stream_copies"] = copies
            row["frac_of_hbm_stream"] = round(compulsory_bytes(c.g) / (t_stream * 1e-3) / 1e9 / hbm_peak, 4)
        if i in read_ms:
            row["read_ceiling_ms"] = round(read_ms[i], 5)
            row["frac_of_read_ceiling"] = round(read_ms[i] / ms, 4)
        per.append(row)
    # dominant kernel: the main kernel of the GEMM with the largest time
    dom = max(range(len(cases)), key=lambda i: statistics.mean(per_gemm_ms[i]))
    dk_ms = statistics.mean(per_kern_ms[dom])
    traffic = load_traffic(cases[dom].g.name)
    if bound_of(cases[dom].g, bf16_peak, hbm_peak) == "tensor":
        roof = {"bound": "tensor", "kernel": f"main kernel of {cases[dom].g.name}",
                "achieved": round(cases[dom].g.flops / (dk_ms * 1e-3) / 1e12, 2), "peak": bf16_peak,
                "unit": "TFLOP/s", "traffic": traffic, "peak_source": f"{peak_src} bf16 dense (burst)"}
    else:
        roof = {"bound": "hbm", "kernel": f"main kernel of {cases[dom].g.name}",
                "achieved": round(compulsory_bytes(cases[dom].g) / (dk_ms * 1e-3) / 1e9, 1), "peak": hbm_peak,
                "unit": "GB/s", "traffic": traffic, "peak_source": f"{peak_src} HBM copy"}
    roof["frac"] = round(roof["achieved"] / roof["peak"], 4)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, args.cpu_seconds)

    value = whole_job_tops(ops, world, gemm_ms)
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(gemm_ms, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": dtype_desc(wl), "data": "synthetic (seeded, workloads.py)",
        "config": config_of(wl, world),
        "per_gemm": per,
        "roofline": roof,
        "e2e": None if e2e_ms is None else {
            "value": round(whole_job_tops(ops, world, e2e_max), 3), "unit": "TOPS",
            "h2d_bytes_per_step": sum(c.h2d for c in cases), "d2h_bytes_per_step": sum(c.d2h for c in cases)},
        "gpu_launches": int(launches),
        "wall_s_timed_region": round(wall, 4),
        "clocks": sampler.summary(),
        "cpu_baseline": cpu,
    }
    return line


def config_of(wl, world):
    """The `config` object of the JSON line, identical in both arms."""
    return {"workload": wl.name, "description": wl.description, "gemms": [g.name for g in wl.gemms],
            "l2": "flushed (512 MiB write) before every timed GEMM; per GEMM also after a clean flush "
                  "(write, then a 256 MiB read)",
            "parallelism": f"replicas x{world}"}


# Source files that determine each kernel family's code: DRAM counters of a
# family are reported only while these files hash to the recorded value.
KERNEL_FAMILIES = {
    "tc": ("gemm_tc.cuh", "gemm_tc2.cuh", "ptx.cuh"),
    "s8tm": ("gemm_s8tm.cu", "ptx.cuh"),
    "skinny": ("gemm_skinny.cu", "ptx.cuh"),
    "tiny": ("gemm_tiny.cu",),
}


def max_over_ranks(values, world, device):
    """Element-wise maximum of per-rank timings over all ranks (a job of
    replicas takes as long as its slowest rank); the values unchanged on one
    rank."""
    vals = torch.tensor(values, dtype=torch.float64, device=device)
    if world > 1:
        torch.distributed.all_reduce(vals, op=torch.distributed.ReduceOp.MAX)
    return vals.tolist()


def whole_job_tops(ops_per_rank, world, ms):
    """Throughput of `world` replicas that each do ops_per_rank operations,
    over the slowest rank's time `ms` (milliseconds), in TOPS."""
    return world * ops_per_rank / (ms * 1e-3) / 1e12


def kernel_source_hash(family: str = "tc") -> str:
    """Hash of one kernel family's sources: counters taken from an older
    kernel are not reported as this kernel's."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_FAMILIES[family]:
        with open(os.path.join(ROOT, "paper_2512_13282_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


_DTYPE_DESC = {"int8": "int8->int32", "int8_int16": "int8->int32->int16", "int8_int8": "int8->int32->int8",
               "bf16": "bf16->fp32->bf16"}


def dtype_desc(wl) -> str:
    """The arithmetic of the workload's GEMMs, e.g. 'int8->int32 and bf16->fp32->bf16'."""
    seen = []
    for g in wl.gemms:
        if _DTYPE_DESC[g.dtype] not in seen:
            seen.append(_DTYPE_DESC[g.dtype])
    return " and ".join(seen)


def compulsory_bytes(g: W.Gemm) -> int:
    """Bytes a GEMM must move at least once: A, B and C (Eq. 6-8 of the
    paper's traffic model with whole-matrix reuse)."""
    e_in = 1 if g.int8_in else 2
    return (g.M * g.K + g.K * g.N) * e_in + g.M * g.N * g.out_bytes


def bound_of(g: W.Gemm, tflops_peak: float, gbs_peak: float) -> str:
    """'tensor' when the flops take longer than the compulsory bytes at the
    measured peaks, else 'hbm'."""
    t_compute = g.flops / (tflops_peak * 1e12)
    t_memory = compulsory_bytes(g) / (gbs_peak * 1e9)
    return "tensor" if t_compute >= t_memory else "hbm"


def load_traffic(name):
    """DRAM bytes (read + write) per launch of the dominant kernel from the
    committed ncu summary (profiles/traffic.json), or None when it was not
    captured for this GEMM or its kernel family's source has changed since."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            d = json.load(f)
        e = d.get("dram_bytes_per_launch", {}).get(name)
        if not e or d.get("kernel_source_hash", {}).get(e["family"]) != kernel_source_hash(e["family"]):
            return None
        return e["bytes"]
    except Exception:
        return None


# ------------------------------------------------------------ CPU oracle

def _oracle_rows(g: W.Gemm, A, B, rows):
    import oracle
    As = np.ascontiguousarray(A[:rows])
    if g.int8_in:
        acc = oracle.gemm_s8(As, B, g.layout)
        if g.dtype != "int8":
            oracle.requantize(acc, g.shift, 8 * g.out_bytes)
    else:
        oracle.gemm_bf16(As, B, g.layout)


def _calibrate_rows(g, A, B, budget):
    """Rows of C the oracle computes in about `budget` seconds (the oracle
    parallelises over rows, so calibrate on one row per thread)."""
    import oracle
    probe = min(g.M, max(1, oracle.num_threads()))
    t0 = time.perf_counter()
    _oracle_rows(g, A, B, probe)
    t1 = time.perf_counter() - t0
    return max(1, min(g.M, int(probe * budget / max(t1, 1e-6))))


def cpu_baseline(wl, seconds):
    """Oracle throughput on whole rows of C of every GEMM of the workload,
    about `seconds` of CPU work in total."""
    import oracle
    oracle.build()
    budget = seconds / len(wl.gemms)
    ops = 0
    t_total = 0.0
    rows_used = []
    for g in wl.gemms:
        A, B = W.make_inputs(g)
        rows = _calibrate_rows(g, A, B, budget)
        t0 = time.perf_counter()
        _oracle_rows(g, A, B, rows)
        dt = time.perf_counter() - t0
        ops += 2 * rows * g.N * g.K
        t_total += dt
        rows_used.append(f"{g.name}:{rows}rows")
    return {"value": round(ops / t_total / 1e12, 6), "unit": "TOPS", "cores": oracle.num_threads(),
            "kind": "oracle", "seconds": round(t_total, 2),
            "sample": "whole rows of C per GEMM (" + ", ".join(rows_used) + ")"}


def run_reference(args, rank, world):
    """The oracle, as it stands, timed on this host's cores on bounded
    samples (whole rows of C) of every GEMM of the workload."""
    import oracle
    oracle.build()
    wl = select(args)
    inputs = [W.make_inputs(g) for g in wl.gemms]
    per_step = args.cpu_seconds_per_step / len(wl.gemms)
    rows = [_calibrate_rows(g, A, B, per_step) for g, (A, B) in zip(wl.gemms, inputs)]
    for _ in range(args.warmup):
        for g, (A, B), r in zip(wl.gemms, inputs, rows):
            _oracle_rows(g, A, B, max(1, r // 8))
    ops, t_total = 0, 0.0
    for _ in range(args.steps):
        for g, (A, B), r in zip(wl.gemms, inputs, rows):
            t0 = time.perf_counter()
            _oracle_rows(g, A, B, r)
            t_total += time.perf_counter() - t0
            ops += 2 * r * g.N * g.K
    value = ops / t_total / 1e12
    sample = "whole rows of C per GEMM per step (" + ", ".join(
        f"{g.name}:{r}rows" for g, r in zip(wl.gemms, rows)) + ")"
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t_total / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": dtype_desc(wl).replace("int32", "int64").replace("fp32", "f64") + " (oracle)",
        "data": "synthetic (seeded, workloads.py)",
        "config": config_of(wl, world),
        "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": oracle.num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }


# ------------------------------------------------------- roofline sweep

SWEEP_DTYPES = (("int8", 0), ("int8_int16", 6), ("int8_int8", 14), ("bf16", 0))


def run_sweep(args, dev):
    """Roofline sweep (Sec. 5.2.3): every size of roofline_sweep_sizes() for
    each output precision and both B layouts.  Operands are the leading
    M*K / K*N elements of 8192^2 seeded master matrices (tight leading
    dimensions).  Each GEMM runs once untimed, then `reps` times, each after
    an L2 flush, between CUDA events; the mean is kept.  A few sampled
    entries of every result are checked against the oracle.  Writes every
    point to `args.sweep` (JSON) and returns the summary line."""
    import oracle
    from paper_2512_13282_gb300 import build as Bld
    from paper_2512_13282_gb300 import gemm as G
    Bld.build()
    G.library()
    oracle.build()
    sizes = W.roofline_sweep_sizes(args.sweep_points)
    big = max(max(m * k, k * n) for m, n, k in sizes)
    hA8 = W.random_int8((big,), 21).reshape(-1)
    hB8 = W.random_int8((big,), 22).reshape(-1)
    hA16 = W.random_bf16((big,), 23).reshape(-1)
    hB16 = W.random_bf16((big,), 24).reshape(-1)
    dA8, dB8 = torch.from_numpy(hA8).to(dev), torch.from_numpy(hB8).to(dev)
    dA16, dB16 = torch.from_numpy(hA16.view(np.int16)).to(dev), torch.from_numpy(hB16.view(np.int16)).to(dev)
    big_c = max(m * n for m, n, _ in sizes)
    dC = torch.empty(big_c * 4, dtype=torch.uint8, device=dev)
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    rng = np.random.default_rng(7)
    peaks, peak_src = load_peaks()
    bf16_peak = float(peaks.get("bf16_tflops", FALLBACK["bf16_tflops"]))
    fns = {"int8": G.gemm_s8s8_s32, "bf16": G.gemm_bf16_f32acc_bf16}
    cdt = {"int8": torch.int32, "int8_int16": torch.int16, "int8_int8": torch.int8, "bf16": torch.int16}
    uuid = str(getattr(torch.cuda.get_device_properties(dev), "uuid", "") or "")
    if uuid and not uuid.startswith("GPU-"):
        uuid = "GPU-" + uuid
    sampler = ClockSampler(uuid)
    sampler.start()
    points, checked, bad = [], 0, 0
    t_start = time.perf_counter()
    for dtype, shift in SWEEP_DTYPES:
        int8 = dtype.startswith("int8")
        dA, dB = (dA8, dB8) if int8 else (dA16, dB16)
        hA, hB = (hA8, hB8) if int8 else (hA16, hB16)
        for layout in (W.B_COL_MAJOR, W.B_ROW_MAJOR):
            for (M, N, K) in sizes:
                g = W.Gemm(M, N, K, dtype, layout, 0, W.I8 if int8 else W.BF, W.I8 if int8 else W.BF, shift)
                ldb = N if layout == W.B_ROW_MAJOR else K
                C = dC.view(cdt[dtype])[:M * N].view(M, N)
                if dtype in ("int8_int16", "int8_int8"):
                    fn = G.gemm_s8s8_s16 if dtype == "int8_int16" else G.gemm_s8s8_s8

                    def launch():
                        return fn(M, N, K, dA, K, dB, ldb, layout, C, N, shift, None)
                else:
                    def launch():
                        return fns[dtype](M, N, K, dA, K, dB, ldb, layout, C, N, None)
                if launch() != 0:
                    raise RuntimeError(f"sweep {g.name}: launch failed")
                evs = []
                for _ in range(args.sweep_reps):
                    flush.fill_(1.0)
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    launch()
                    b.record(stream)
                    evs.append((a, b))
                r = np.concatenate([rng.integers(0, M, 3), [M - 1]])
                c = np.concatenate([rng.integers(0, N, 3), [N - 1]])
                got = C[torch.from_numpy(r).to(dev), torch.from_numpy(c).to(dev)].cpu().numpy()
                ms = statistics.mean(x.elapsed_time(y) for x, y in evs)
                Ah = hA[:M * K].reshape(M, K)
                Bh = hB[:K * N].reshape((K, N) if layout == W.B_ROW_MAJOR else (N, K))
                if int8:
                    want = oracle.gemm_s8_entries(Ah, Bh, layout, r, c)
                    if dtype != "int8":
                        want = oracle.requantize(want, shift, 8 * g.out_bytes)
                    nbad = int(np.sum(got.astype(np.int64) != want))
                else:
                    ref, mag = oracle.gemm_bf16_entries(Ah, Bh, layout, r, c)
                    nbad = int(np.sum(~oracle.bf16_within_bound(got.view(np.uint16), ref, mag)))
                checked += r.size
                bad += nbad
                tops = g.flops / (ms * 1e-3) / 1e12
                points.append({"dtype": dtype, "layout": "col" if layout == W.B_COL_MAJOR else "row",
                               "M": M, "N": N, "K": K, "ms": round(ms, 5), "tops": round(tops, 2),
                               "ari": round(g.flops / compulsory_bytes(g), 1), "mismatches": nbad})
    torch.cuda.synchronize()
    sampler.stop()
    wall = time.perf_counter() - t_start

    summary = {}
    for dtype, _ in SWEEP_DTYPES:
        per = {}
        for lay in ("col", "row"):
            v = [p for p in points if p["dtype"] == dtype and p["layout"] == lay]
            t = np.array([p["tops"] for p in v])
            hi = np.array([p["tops"] for p in v if p["ari"] > 1000])
            best = max(v, key=lambda p: p["tops"])
            per[lay] = {"points": len(v), "mean_tops": round(float(t.mean()), 1),
                        "median_tops": round(float(np.median(t)), 1), "max_tops": best["tops"],
                        "max_at": [best["M"], best["N"], best["K"]],
                        "mean_frac_of_bf16_peak": round(float(t.mean()) / bf16_peak, 4),
                        "ari_gt_1000": {"points": int(hi.size),
                                        "mean_tops": round(float(hi.mean()), 1) if hi.size else None,
                                        "cov": round(float(hi.std() / hi.mean()), 4) if hi.size else None}}
        per["col_over_row_mean_pct"] = round(100.0 * (per["col"]["mean_tops"] / per["row"]["mean_tops"] - 1), 2)
        summary[dtype] = per
    with open(args.sweep, "w") as f:
        json.dump({"sizes_rule": W.roofline_sweep_sizes.__doc__.split("\n")[0], "points": points}, f)
    return {"metric": "roofline sweep: TOPS per GEMM size, B column- and row-major", "unit": "TOPS",
            "sizes_per_layout": len(sizes), "gemms": len(points), "reps": args.sweep_reps,
            "peak_bf16_tflops": bf16_peak, "peak_source": peak_src, "summary": summary,
            "parity": {"entries_checked": checked, "mismatches": bad}, "clocks": sampler.summary(),
            "wall_s": round(wall, 1), "points_file": args.sweep}


def parse_shape(text: str) -> W.Gemm:
    """One GEMM from 'DTYPE:MxNxK:LAYOUT', e.g. 'int8:5120x5120x5120:row'
    (DTYPE int8, int8_int16, int8_int8 or bf16; LAYOUT row or col): int8
    operands uniform on [-128, 127], bf16 N(0, 1), seed 0, shift 7 for the
    requantised outputs."""
    try:
        dtype, dims, lay = text.split(":")
        M, N, K = (int(x) for x in dims.lower().split("x"))
    except ValueError:
        raise SystemExit(f"--shape wants DTYPE:MxNxK:LAYOUT, got {text!r}")
    if dtype not in ("int8", "int8_int16", "int8_int8", "bf16") or lay not in ("row", "col") or min(M, N, K) < 1:
        raise SystemExit(f"--shape: unknown dtype / layout or empty size in {text!r}")
    d = W.BF if dtype == "bf16" else W.I8
    return W.Gemm(M, N, K, dtype, W.B_ROW_MAJOR if lay == "row" else W.B_COL_MAJOR, 0, d, d,
                  7 if dtype in ("int8_int16", "int8_int8") else 0)


def select(args) -> W.Workload:
    """The workload (or the one GEMM of --shape), optionally narrowed to the
    GEMMs named by --gemm."""
    if args.shape:
        g = parse_shape(args.shape)
        return W.Workload("shape", f"one GEMM {g.name}, seed 0", (g,))
    wl = W.WORKLOADS[args.workload]
    if not args.gemm:
        return wl
    keep = tuple(g for g in wl.gemms if g.name in args.gemm)
    if not keep:
        raise SystemExit(f"--gemm matched nothing in {wl.name}: {[g.name for g in wl.gemms]}")
    return W.Workload(wl.name, wl.description + " (subset: " + ", ".join(g.name for g in keep) + ")", keep)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="all_configs", choices=sorted(W.WORKLOADS))
    ap.add_argument("--shape", metavar="DTYPE:MxNxK:LAYOUT",
                    help="time one GEMM of this shape instead of a workload, e.g. int8:5120x5120x5120:row")
    ap.add_argument("--gemm", action="append", default=[],
                    help="run only this GEMM of the workload (repeatable), e.g. bf16_4096x4096x4096_Bcol")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-stream", action="store_true", help="skip the back-to-back pass of the HBM-bound GEMMs")
    ap.add_argument("--cpu-seconds", type=float, default=30.0)
    ap.add_argument("--cpu-seconds-per-step", type=float, default=6.0)
    ap.add_argument("--sweep", metavar="OUT.json",
                    help="run the roofline sweep instead (every point written to OUT.json)")
    ap.add_argument("--sweep-points", type=int, default=420)
    ap.add_argument("--sweep-reps", type=int, default=3)
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, rank, world)), flush=True)
        return

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if args.sweep:
        if rank == 0:
            print(json.dumps(run_sweep(args, dev)), flush=True)
        return
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=dev)
    line = run_ours(args, rank, world, dev)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()

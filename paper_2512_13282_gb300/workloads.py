"""Seeded synthetic inputs for the GEMM C = A.B (no GEMM arithmetic here).

The paper measures on synthetic matrices of chosen sizes only (Sec. 5.2.3:
sweeps of GEMM sizes up to 8K, B row- and column-major); there is no dataset.
The workloads below are those sizes, layouts and value distributions.

Recipe, per GEMM instance: a fresh CPU ``torch.Generator`` seeded with the
workload's seed draws A, then B.  int8 entries come from ``torch.randint``
(uniform, inclusive bounds); bf16 entries from ``torch.randn`` in float32,
scaled, then rounded to bfloat16 by torch (nearest-even).  Arrays are returned
as numpy: int8, or uint16 bf16 bit patterns.  A is row-major M x K; B is
row-major K x N (layout 0) or column-major, i.e. stored N x K (layout 1).
Both sides of every comparison -- the CUDA library and the oracle -- receive
the same arrays from here.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

B_ROW_MAJOR = 0
B_COL_MAJOR = 1


@dataclass(frozen=True)
class Dist:
    """Entry distribution: int8 uniform on [lo, hi], or bf16 of scale*N(0,1)."""
    kind: str            # "int8" or "bf16"
    lo: int = -128
    hi: int = 127
    scale: float = 1.0


@dataclass(frozen=True)
class Gemm:
    M: int
    N: int
    K: int
    dtype: str           # "int8" (int32 C), "int8_int16" / "int8_int8" (requantised C) or "bf16"
    layout: int
    seed: int
    a: Dist
    b: Dist
    shift: int = 0       # right shift of the requantised int8 outputs

    @property
    def int8_in(self) -> bool:
        return self.dtype.startswith("int8")

    @property
    def out_bytes(self) -> int:
        """Bytes per element of C."""
        return {"int8": 4, "int8_int16": 2, "int8_int8": 1, "bf16": 2}[self.dtype]

    @property
    def flops(self) -> int:
        return 2 * self.M * self.N * self.K

    @property
    def name(self) -> str:
        lay = "Bcol" if self.layout == B_COL_MAJOR else "Brow"
        return f"{self.dtype}_{self.M}x{self.N}x{self.K}_{lay}"


@dataclass(frozen=True)
class Workload:
    name: str
    description: str
    gemms: tuple = field(default_factory=tuple)


I8 = Dist("int8", -128, 127)
I8_HALF = Dist("int8", -64, 63)
BF = Dist("bf16", scale=1.0)
BF_01 = Dist("bf16", scale=0.1)
BF_002 = Dist("bf16", scale=0.02)


def _both(M, N, K, layout, seed, ia=I8, ib=I8, ba=BF, bb=BF):
    return (Gemm(M, N, K, "int8", layout, seed, ia, ib),
            Gemm(M, N, K, "bf16", layout, seed, ba, bb))


WORKLOADS = {
    "int8_square_256": Workload(
        "int8_square_256",
        "int8 GEMM 256^3, A and B row-major, uniform [-128,127], seed 0",
        (Gemm(256, 256, 256, "int8", B_ROW_MAJOR, 0, I8, I8),)),
    "square_sweep_512_4096": Workload(
        "square_sweep_512_4096",
        "square GEMMs M=N=K in {512,1024,2048,4096}, int8 uniform [-128,127] and "
        "bf16 N(0,1); A row-major, B column-major (N x K), seed 1",
        tuple(g for s in (512, 1024, 2048, 4096) for g in _both(s, s, s, B_COL_MAJOR, 1))),
    "square_8192": Workload(
        "square_8192",
        "square GEMM 8192^3, int8 uniform [-128,127] and bf16 0.1*N(0,1); "
        "A and B row-major, seed 2",
        _both(8192, 8192, 8192, B_ROW_MAJOR, 2, ba=BF_01, bb=BF_01)),
    "transformer_projections": Workload(
        "transformer_projections",
        "projection GEMMs, M in {128,2048}, (K,N) in {(4096,4096),(4096,11008),"
        "(11008,4096),(4096,12288)}; A int8 [-128,127] or bf16 N(0,1), B int8 "
        "[-64,63] or bf16 0.02*N(0,1); B column-major (N x K), seed 3",
        tuple(g for M in (128, 2048)
              for (K, N) in ((4096, 4096), (4096, 11008), (11008, 4096), (4096, 12288))
              for g in _both(M, N, K, B_COL_MAJOR, 3, ib=I8_HALF, bb=BF_002))),
    "reduced_precision_outputs": Workload(
        "reduced_precision_outputs",
        "int8 GEMMs with outputs reduced to int16 (right shift 6) and int8 (right shift 14), "
        "M=N=K in {4096, 8192}, uniform [-128,127]; A row-major, B column-major (N x K), seed 1",
        tuple(Gemm(s, s, s, dt, B_COL_MAJOR, 1, I8, I8, sh) for s in (4096, 8192)
              for dt, sh in (("int8_int16", 6), ("int8_int8", 14)))),
    "irregular_skinny": Workload(
        "irregular_skinny",
        "irregular and skinny shapes (1000,1500,3000), (16,4096,4096), "
        "(1,11008,4096), (3072,2560,777), (8192,64,8192); int8 [-128,127] and "
        "bf16 N(0,1); A and B row-major, seed 4",
        tuple(g for (M, N, K) in ((1000, 1500, 3000), (16, 4096, 4096), (1, 11008, 4096),
                                  (3072, 2560, 777), (8192, 64, 8192))
              for g in _both(M, N, K, B_ROW_MAJOR, 4))),
}


# The five benchmark configurations in one step, in the order listed above.
BENCHMARK_CONFIGS = ("int8_square_256", "square_sweep_512_4096", "square_8192", "transformer_projections",
                     "irregular_skinny")
WORKLOADS["all_configs"] = Workload(
    "all_configs",
    "every GEMM of the five benchmark configurations: int8 256^3 (seed 0); square sweep 512..4096 "
    "both paths (seed 1); 8192^3 both paths (seed 2); transformer projections (seed 3); irregular "
    "and skinny shapes (seed 4)",
    tuple(g for name in BENCHMARK_CONFIGS for g in WORKLOADS[name].gemms))


def roofline_sweep_sizes(points: int = 420, seed: int = 5, step: int = 256, largest: int = 8192):
    """(M, N, K) triples of the roofline sweep: the paper sweeps more than
    400 sizes per B layout, each a multiple of the native GEMM size, up to
    8K, favouring no dimension (Sec. 5.2.3).  Here the native size is 256
    (the CTA-pair tile); M, N and K are drawn independently as step * j,
    j in 1 .. largest/step with probability proportional to 1/j (uniform in
    log size, so small and large arithmetic intensities are both well
    covered), without repeated triples, from numpy's default_rng(seed)."""
    rng = np.random.default_rng(seed)
    j = np.arange(1, largest // step + 1)
    prob = (1.0 / j) / np.sum(1.0 / j)
    seen, out = set(), []
    while len(out) < points:
        t = tuple(int(step * x) for x in rng.choice(j, 3, p=prob))
        if t not in seen:
            seen.add(t)
            out.append(t)
    return out


def _draw(gen: torch.Generator, rows: int, cols: int, d: Dist) -> np.ndarray:
    if d.kind == "int8":
        t = torch.randint(d.lo, d.hi + 1, (rows, cols), generator=gen, dtype=torch.int8)
        return t.numpy()
    t = torch.randn((rows, cols), generator=gen, dtype=torch.float32)
    if d.scale != 1.0:
        t = t * d.scale
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def make_inputs(g: Gemm):
    """(A, B) for one GEMM instance: A is M x K; B is K x N (layout 0) or
    N x K (layout 1)."""
    gen = torch.Generator().manual_seed(g.seed)
    A = _draw(gen, g.M, g.K, g.a)
    if g.layout == B_ROW_MAJOR:
        B = _draw(gen, g.K, g.N, g.b)
    else:
        B = _draw(gen, g.N, g.K, g.b)
    return A, B


def random_int8(shape, seed: int, lo: int = -128, hi: int = 127) -> np.ndarray:
    gen = torch.Generator().manual_seed(seed)
    return torch.randint(lo, hi + 1, tuple(shape), generator=gen, dtype=torch.int8).numpy()


def random_bf16(shape, seed: int, scale: float = 1.0) -> np.ndarray:
    gen = torch.Generator().manual_seed(seed)
    t = torch.randn(tuple(shape), generator=gen, dtype=torch.float32) * scale
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def integer_bf16(shape, seed: int, lo: int = -8, hi: int = 8) -> np.ndarray:
    """bf16 bit patterns of small integers in [lo, hi] (exact in bf16)."""
    gen = torch.Generator().manual_seed(seed)
    t = torch.randint(lo, hi + 1, tuple(shape), generator=gen, dtype=torch.int32).to(torch.float32)
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)

"""Seeded synthetic inputs for the permutation-group Allreduce workloads.

Shared by the tests, ``bench.py`` and ``__graft_entry__.smoke()``: the same tensors go
to the CUDA library and (copied to the host) to the CPU oracle.  This module holds no
part of the Allreduce itself -- only workload shapes and random number generation.

The workloads follow the message sizes the paper experiments with (Kolmakov & Zhang,
arXiv 2004.09362, Sec. "Experimental results"): the 425-byte average Allreduce size and
P = 127 processes, plus a gradient-bucket-shaped large case.  No dataset is involved.
"""

from __future__ import annotations

from dataclasses import dataclass

import torch

__all__ = ["Workload", "WORKLOADS", "rank_inputs", "batched_inputs", "TORCH_DTYPE"]

TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16, "i32": torch.int32}


@dataclass(frozen=True)
class Workload:
    name: str
    P: int
    n: int                 # elements per rank
    dtype: str             # "f32" | "bf16" | "i32"
    dist: tuple            # ("uniform", lo, hi) | ("normal", mean, std) | ("int", lo, hi)
    ops: tuple
    steps: tuple           # step counts exercised (L..2L)
    seed: int


def _L(P: int) -> int:
    L = 0
    while (1 << L) < P:
        L += 1
    return L


WORKLOADS = {
    # P=5, 1024 fp32 per rank, U[-1,1]; latency-optimal (3 steps) and every other S.
    "p5_f32": Workload("p5_f32", 5, 1024, "f32", ("uniform", -1.0, 1.0), ("sum",),
                       (3, 4, 5, 6), 1234),
    "p5_i32": Workload("p5_i32", 5, 1024, "i32", ("int", -1000, 1000), ("sum", "max", "min"),
                       (3, 4, 5, 6), 1234),
    # P=8 (power of two), 1 MiB fp32 per rank, U[-1,1], S = 3..6.
    "p8_1mib_f32": Workload("p8_1mib_f32", 8, 262144, "f32", ("uniform", -1.0, 1.0),
                            ("sum",), (3, 4, 5, 6), 1235),
    # P=24, 64 MiB fp32 per rank (gradient-bucket shaped), N(0, 1e-3), bandwidth-optimal.
    "p24_64mib_f32": Workload("p24_64mib_f32", 24, 16777216, "f32", ("normal", 0.0, 1e-3),
                              ("sum",), (10,), 1237),
    # P=127 (prime), 8 MiB bf16 per rank, N(0,1), fp32 accumulation, S = 7..14.
    "p127_8mib_bf16": Workload("p127_8mib_bf16", 127, 4194304, "bf16", ("normal", 0.0, 1.0),
                               ("sum",), tuple(range(7, 15)), 1238),
}

# 65536 independent Allreduces of 106 fp32 elements per rank (~425 bytes), half with
# P=6 and half with P=7, N(0,1), sum and max, latency-optimal schedule.
BATCHED = {"count": 65536, "Ps": (6, 7), "n": 106, "dtype": "f32",
           "dist": ("normal", 0.0, 1.0), "ops": ("sum", "max"), "seed": 1236}


def _fill(shape, dist, dtype: str, gen: torch.Generator, device) -> torch.Tensor:
    kind = dist[0]
    if kind == "int":
        lo, hi = int(dist[1]), int(dist[2])
        return torch.randint(lo, hi + 1, shape, generator=gen, device=device, dtype=torch.int32)
    if kind == "uniform":
        lo, hi = float(dist[1]), float(dist[2])
        t = torch.rand(shape, generator=gen, device=device, dtype=torch.float32)
        t = t * (hi - lo) + lo
    elif kind == "normal":
        mean, std = float(dist[1]), float(dist[2])
        t = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        t = t * std + mean
    else:
        raise ValueError(dist)
    return t.to(TORCH_DTYPE[dtype])


def rank_inputs(P: int, n: int, dtype: str, dist, seed: int, device="cpu") -> torch.Tensor:
    """A [P, n] tensor: row x is rank x's input vector."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    return _fill((P, n), dist, dtype, gen, device)


def batched_inputs(count: int, Ps, n: int, dtype: str, dist, seed: int, device="cpu"):
    """Inputs for ``count`` independent Allreduces: the first count/len(Ps) instances
    use Ps[0] ranks, the next Ps[1], ...  Returns (flat tensor, list of (P, offset))
    with each instance stored as a contiguous [P, n] row-major slab."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    per = count // len(Ps)
    layout = []
    off = 0
    for gi, P in enumerate(Ps):
        cnt = per if gi < len(Ps) - 1 else count - per * (len(Ps) - 1)
        for _ in range(cnt):
            layout.append((P, off))
            off += P * n
    flat = _fill((off,), dist, dtype, gen, device)
    return flat, layout

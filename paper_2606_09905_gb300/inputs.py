"""Seeded synthetic inputs shared by the tests, the bench and the smoke check.

This module holds no arithmetic of the method: it only draws operands.  Both
the CUDA path and the CPU oracle consume the tensors it returns, which is the
one thing the two sides share.

Recipe: a CPU ``torch.Generator`` seeded with ``seed``; integer operands are
i.i.d. uniform on the inclusive range [lo, hi] (``torch.randint(lo, hi + 1)``),
FP32 operands are i.i.d. N(0, 1) (``torch.randn``).  A, B (or x, w, or Q, K, V)
are drawn in that order from the one generator.  Tensors come back on the CPU,
contiguous; callers move them to the device.

The paper (Table 1, Table 2) names its workloads only by size and data type;
``WORKLOADS`` gives the synthetic shapes and value ranges used in their place.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


def int_uniform(shape, lo: int, hi: int, gen: torch.Generator,
                dtype: torch.dtype = torch.int16) -> torch.Tensor:
    return torch.randint(lo, hi + 1, tuple(shape), generator=gen, dtype=dtype)


def normal(shape, gen: torch.Generator) -> torch.Tensor:
    return torch.randn(tuple(shape), generator=gen, dtype=torch.float32)


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator()
    g.manual_seed(int(seed))
    return g


def gemm_case(M: int, N: int, K: int, lo: int, hi: int, seed: int,
              dtype: torch.dtype = torch.int16):
    """Row-major A (M x K) and B (K x N)."""
    g = _gen(seed)
    return int_uniform((M, K), lo, hi, g, dtype), int_uniform((K, N), lo, hi, g, dtype)


def conv_case(n: int, c: int, h: int, w: int, k: int, r: int, s: int,
              lo: int, hi: int, seed: int, dtype: torch.dtype = torch.int16):
    """NCHW input x and KCRS weights."""
    g = _gen(seed)
    return int_uniform((n, c, h, w), lo, hi, g, dtype), int_uniform((k, c, r, s), lo, hi, g, dtype)


def conv_case_f32(n, c, h, w, k, r, s, seed):
    g = _gen(seed)
    return normal((n, c, h, w), g), normal((k, c, r, s), g)


def attn_case(L: int, d: int, lo: int, hi: int, seed: int,
              dtype: torch.dtype = torch.int16, heads: int = 0):
    """Q, K, V, each L x d row-major; heads >= 1 gives heads x L x d."""
    g = _gen(seed)
    shape = (L, d) if heads == 0 else (heads, L, d)
    return tuple(int_uniform(shape, lo, hi, g, dtype) for _ in range(3))


def attn_case_f32(L: int, d: int, seed: int, heads: int = 0):
    g = _gen(seed)
    shape = (L, d) if heads == 0 else (heads, L, d)
    return tuple(normal(shape, g) for _ in range(3))


def lenet_case(batch: int, seed: int, x_hi: int = 255, w_mag: int = 7):
    """LeNet-shaped INT32 pipeline operands: images N x 1 x 32 x 32 uniform in
    [0, x_hi] (pixels), then w1 6x1x5x5, w2 16x6x5x5, w3 400x120, w4 120x84,
    w5 84x10, each uniform in [-w_mag, w_mag]; all int32."""
    g = _gen(seed)
    x = int_uniform((batch, 1, 32, 32), 0, x_hi, g, torch.int32)
    shapes = ((6, 1, 5, 5), (16, 6, 5, 5), (400, 120), (120, 84), (84, 10))
    ws = tuple(int_uniform(sh, -w_mag, w_mag, g, torch.int32) for sh in shapes)
    return (x,) + ws


@dataclass(frozen=True)
class Workload:
    name: str
    op: str                     # "gemm" | "conv" | "attn"
    shape: dict
    lo: int = 0
    hi: int = 0
    note: str = ""
    extra: dict = field(default_factory=dict)


# The five workload families (Table 1 GEMM sizes; Table 2 conv / attention
# rows; the 8192^3 case for the tensor-core roofline).
WORKLOADS = {
    "gemm256": Workload("gemm256", "gemm", dict(M=256, N=256, K=256), -1023, 1023,
                        "INT16 GEMM 256^3, also run as INT32 operands"),
    "gemm512": Workload("gemm512", "gemm", dict(M=512, N=512, K=512), -1023, 1023),
    "gemm768": Workload("gemm768", "gemm", dict(M=768, N=768, K=768), -1023, 1023),
    "gemm1024": Workload("gemm1024", "gemm", dict(M=1024, N=1024, K=1024), -1023, 1023),
    "gemm2048": Workload("gemm2048", "gemm", dict(M=2048, N=2048, K=2048), -1023, 1023),
    "gemm4096x64x1024": Workload("gemm4096x64x1024", "gemm", dict(M=4096, N=64, K=1024),
                                 -1023, 1023, "skinny attention-like shape"),
    "conv": Workload("conv", "conv", dict(n=8, c=64, h=56, w=56, k=128, r=3, s=3,
                                          stride=1, pad=1), -255, 255),
    "attn": Workload("attn", "attn", dict(L=1024, d=64), -7, 7),
    "gemm8192": Workload("gemm8192", "gemm", dict(M=8192, N=8192, K=8192), -500, 500,
                         "large INT16 GEMM, K*500^2 < 2^31"),
}

"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle
checks.  Holds none of the method's arithmetic: only random draws and casts.

Recipe: q, k, v, dout ~ N(0, 1) drawn in fp32 from a torch CPU generator,
then cast to the I/O dtype; per-layer tensors use seed * 1000 + layer; the
learned schedule's theta_l ~ N(0, 0.5) (standard deviation 0.5) per layer.
"""
from __future__ import annotations

import torch


def layer_seed(seed: int, layer: int) -> int:
    return seed * 1000 + layer


def normal(shape, seed: int, dtype=torch.float32, device="cpu") -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    x = torch.randn(*shape, generator=g, dtype=torch.float32)
    return x.to(dtype=dtype, device=device)


def qkv(B: int, H: int, T: int, seed: int, dtype=torch.float32, Hkv=None, D: int = 64, device="cpu"):
    """q [B,H,T,D], k, v [B,Hkv,T,D]; three independent streams of one seed."""
    Hkv = Hkv or H
    q = normal((B, H, T, D), seed * 3 + 0, dtype, device)
    k = normal((B, Hkv, T, D), seed * 3 + 1, dtype, device)
    v = normal((B, Hkv, T, D), seed * 3 + 2, dtype, device)
    return q, k, v


def dout(B: int, H: int, T: int, seed: int, dtype=torch.float32, D: int = 64, device="cpu"):
    return normal((B, H, T, D), seed * 7 + 5, dtype, device)


def theta_learned(L: int, seed: int, std: float = 0.5):
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed) * 11 + 3)
    return (torch.randn(L, generator=g, dtype=torch.float64) * std).tolist()


def device_normal_(t: torch.Tensor, seed: int) -> torch.Tensor:
    """Fill a device tensor with N(0,1) from a seeded device generator (bench
    inputs too large to draw on the host; not used for oracle comparisons)."""
    g = torch.Generator(device=t.device)
    g.manual_seed(int(seed))
    if t.dtype == torch.float32:
        t.normal_(generator=g)
    else:
        tmp = torch.empty(t.shape, dtype=torch.float32, device=t.device)
        tmp.normal_(generator=g)
        t.copy_(tmp)
    return t

"""GPU parity of the RoPE prologue: the rotated keys (fp16 rows that the
forward keeps for the backward) against the rotation written as complex
multiplication (numpy, fp64), for both tile shapes the prologue picks (8
positions x 32 heads when those tiles still give two blocks per SM, else x 16)
and for ragged ends (T and the number of kv-head rows not multiples of a tile).

Bar: |k~ - ref| <= 2^-11 |ref| + 4e-6 (|k_m| + |k_m+32|) + 1e-7 per entry --
fp16 round-to-nearest (11 significant bits) of a rotation whose angle is the
fixed-point phase (exact modulo one turn) evaluated in fp32 (cos and sin to
~1e-6 absolute).
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs
from tests.independent_forms import rope_complex_np

pytestmark = pytest.mark.gpu

# (B, H, Hkv, T): kv-head rows B * Hkv and positions T
CASES = [
    (16, 8, 8, 1024),    # 512 tiles of 32 heads: the 32-head form on a 152-SM GPU
    (17, 8, 8, 1020),    # 32-head form with a partial head tile (136 rows) and a partial position tile
    (5, 8, 8, 1000),     # 16-head form, 40 rows: a partial head tile
    (2, 6, 3, 333),      # 16-head form, 6 rows (under one tile), ragged T
    (1, 2, 1, 7),        # a single partial tile
]


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}" for c in CASES])
def test_rotated_keys_match_the_rotation(case):
    Bn, H, Hkv, T = case
    q, k, v = inputs.qkv(Bn, H, T, seed=7 * T + Bn, dtype=torch.bfloat16, Hkv=Hkv)
    qc, kc, vc = q.cuda(), k.cuda(), v.cuda()
    f = fa.base("fib", 15)
    rk = fa.rotated_k_like(kc)
    fa.fwd(qc, kc, vc, 0.9, f, 8, rotated_k=rk)
    torch.cuda.synchronize()
    assert rk.dtype == torch.float16
    got = rk.cpu().to(torch.float64).numpy().reshape(Bn * Hkv, T, 64)
    kf = k.to(torch.float64).numpy().reshape(Bn * Hkv, T, 64)
    ref = rope_complex_np(kf)
    pair = np.abs(kf[..., :32]) + np.abs(kf[..., 32:])
    bound = 2.0 ** -11 * np.abs(ref) + 4e-6 * np.concatenate([pair, pair], axis=-1) + 1e-7
    err = np.abs(got - ref)
    assert np.all(err <= bound), float(np.max(err - bound))

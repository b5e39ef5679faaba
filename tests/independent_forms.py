"""Independent restatements used to pin the oracle (tests only).

These are written differently from ``oracle/fibattn_oracle.c`` on purpose, so a
slip in one is unlikely to be repeated in the other:

* RoPE is applied as a complex multiplication z_m * exp(i * pos * theta_m) on
  the pairs (x_m, x_{m+D/2}), with theta_m = exp(-(2m/D) ln base).
* The attended set of Section 2 is built as an explicit T x T boolean mask
  (integer distances) or as a per-query interpolation matrix G (continuous
  distances), and attention is computed with whole-matrix operations.
"""
from __future__ import annotations

import math

import numpy as np
import torch


# ---------------------------------------------------------------- RoPE ----

def rope_complex_np(x: np.ndarray, base: float = 1e4) -> np.ndarray:
    """x [..., T, D] -> rotated at positions 0..T-1 via complex multiplication."""
    T, D = x.shape[-2], x.shape[-1]
    half = D // 2
    theta = np.exp(-(2.0 * np.arange(half) / D) * math.log(base))
    ang = np.arange(T)[:, None] * theta[None, :]
    z = x[..., :half] + 1j * x[..., half:]
    z = z * np.exp(1j * ang)
    return np.concatenate([z.real, z.imag], axis=-1)


def rope_complex_torch(x: torch.Tensor, base: float = 1e4) -> torch.Tensor:
    T, D = x.shape[-2], x.shape[-1]
    half = D // 2
    theta = torch.exp(-(2.0 * torch.arange(half, dtype=torch.float64) / D) * math.log(base))
    ang = torch.arange(T, dtype=torch.float64)[:, None] * theta[None, :]
    c, s = torch.cos(ang), torch.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return torch.cat([a * c - b * s, a * s + b * c], dim=-1)


# ------------------------------------------------- dense boolean mask ----

def bool_mask(T: int, W: int, dist_int, dedup: bool = True) -> np.ndarray:
    """mask[i, j] = True when key j is attended by query i for integer rung
    distances (the fused boolean-mask form of Section 2, "Implementation note")."""
    i = np.arange(T)[:, None]
    j = np.arange(T)[None, :]
    delta = i - j
    m = (delta >= 0) & (delta <= W)
    for dk in dist_int:
        dk = int(dk)
        if dedup and dk <= W:
            continue
        m |= (delta == dk)
    return m


def masked_attention_np(q, k, v, mask, scale, base=1e4, kv_group=1):
    """Dense softmax attention with an explicit boolean mask, fp64.
    q [B,H,T,D]; k, v [B,Hkv,T,D]; mask [T,T]."""
    qt = rope_complex_np(q, base)
    kt = rope_complex_np(k, base)
    kt = np.repeat(kt, kv_group, axis=1)
    vv = np.repeat(v, kv_group, axis=1)
    s = scale * np.einsum("bhid,bhjd->bhij", qt, kt)
    s = np.where(mask[None, None], s, -np.inf)
    mx = s.max(axis=-1, keepdims=True)
    e = np.exp(s - mx)
    l = e.sum(axis=-1, keepdims=True)
    p = e / l
    o = np.einsum("bhij,bhjd->bhid", p, vv)
    lse = (mx + np.log(l))[..., 0]
    return o, lse


# ------------------------------------------ interpolation-matrix form ----

def interp_matrix(T: int, W: int, d: torch.Tensor, dedup: bool = True):
    """Build G [T, S, T] (S = W+1+K) and a slot-validity mask [T, S].

    Row (i, slot) of G holds the interpolation weights that read the slot's
    key from the key rows: a window slot t has a single 1 at column i-t; rung
    k has (1-w_k) at column i-floor(d_k) and w_k at column i-floor(d_k)-1
    (dropped when that column is -1).  w_k keeps its autograd graph to d."""
    K = d.shape[0]
    S = W + 1 + K
    s0 = torch.floor(d).detach()
    w = d - s0
    valid = torch.zeros(T, S, dtype=torch.bool)
    idx_i, idx_s, idx_j, vals = [], [], [], []
    one = torch.ones((), dtype=torch.float64)
    for i in range(T):
        for t in range(W + 1):
            if i - t >= 0:
                valid[i, t] = True
                idx_i.append(i); idx_s.append(t); idx_j.append(i - t); vals.append(one)
    for kk in range(K):
        dk = float(d[kk].detach())
        if dedup and dk <= W:
            continue
        sk = int(s0[kk])
        for i in range(T):
            if dk > i:
                continue
            valid[i, W + 1 + kk] = True
            idx_i.append(i); idx_s.append(W + 1 + kk); idx_j.append(i - sk); vals.append(1.0 - w[kk])
            if i - sk - 1 >= 0:
                idx_i.append(i); idx_s.append(W + 1 + kk); idx_j.append(i - sk - 1); vals.append(w[kk])
    G = torch.zeros(T, S, T, dtype=torch.float64)
    G = G.index_put((torch.tensor(idx_i), torch.tensor(idx_s), torch.tensor(idx_j)),
                    torch.stack(vals), accumulate=True)
    return G, valid


def matrix_attention_torch(q, k, v, W, d, scale, base=1e4, dedup=True, kv_group=1):
    """Interpolated sparse attention as whole-matrix torch ops (fp64, autograd).
    q [B,H,T,D]; k, v [B,Hkv,T,D]; d [K] (may require grad through alpha)."""
    T = q.shape[-2]
    G, valid = interp_matrix(T, W, d, dedup)
    qt = rope_complex_torch(q, base)
    kt = rope_complex_torch(k, base)
    kt = kt.repeat_interleave(kv_group, dim=1)
    vv = v.repeat_interleave(kv_group, dim=1)
    keys = torch.einsum("isj,bhjd->bhisd", G, kt)
    vals = torch.einsum("isj,bhjd->bhisd", G, vv)
    s = scale * torch.einsum("bhid,bhisd->bhis", qt, keys)
    s = s.masked_fill(~valid[None, None], float("-inf"))
    p = torch.softmax(s, dim=-1)
    o = torch.einsum("bhis,bhisd->bhid", p, vals)
    lse = torch.logsumexp(s, dim=-1)
    return o, lse

"""GPU parity at input magnitudes away from unit scale.

Training in bf16 autocast (Section 3, "Model and training") hands the
attention backward upstream gradients far below 1: per-token dO of 1e-5 to
1e-8 is common.  bf16 carries fp32's exponent range, so the library must not
lose such gradients inside its own 16-bit operands.  These cases scale dO by
2^-16, 2^-20 and 2^-24 and compare every gradient with the fp64 oracle on the
same (scaled, bf16) inputs, per tensor relative to the largest reference
magnitude -- with no absolute floor, since every reference here is small.

A second case moves the operand range without changing the scores: q scaled
by 2^6 and k by 2^-6 leaves every score q~.k~ as it is, so the bars stay
those of unit inputs while the rotated rows and the gradients dk (x 2^6) and
dq (x 2^-6) sit far from unit scale.  (Scaling q and k both up multiplies the
scores: with 16-bit rotated operands the score error grows with the score
itself, and a softmax of scores in the thousands is decided by near-ties.)
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs
from tests.test_gpu_parity import NTHREADS, _f64, bf16_out_tol

pytestmark = pytest.mark.gpu

GRAD_TOL = 3e-2


def _rel(a, ref):
    return float(np.max(np.abs(a - ref)) / np.max(np.abs(ref)))


def _reference(q, k, v, g, alpha, f, W):
    a32 = float(np.float32(alpha))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    ro, rl = O.forward(_f64(q), _f64(k), _f64(v), W, d, nthreads=NTHREADS)
    rq, rk, rv, rdd = O.backward(_f64(q), _f64(k), _f64(v), _f64(g), W, d, nthreads=NTHREADS)
    _, rth = O.dtheta(a32, f.astype(np.float64), rdd)
    return ro, rl, rq, rk, rv, rdd, rth


def _run(q, k, v, g, alpha, f, W, path):
    """path: "mma" (forward output given, scores recomputed), "residuals" (the
    training path: rotated keys and residuals kept from the forward), "gather"."""
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), g.cuda()
    if path == "residuals":
        rk = fa.rotated_k_like(kc)
        res = fa.residuals_like(qc, W, len(f))
        out, lse = fa.fwd(qc, kc, vc, alpha, f, W, rotated_k=rk, residuals=res)
        grads = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, out=out, rotated_k=rk, residuals=res)
    else:
        out, lse = fa.fwd(qc, kc, vc, alpha, f, W)
        grads = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, kernel=path, out=None if path == "gather" else out)
    torch.cuda.synchronize()
    return out, lse, grads


def _check(q, k, v, g, alpha, f, W, path):
    out, lse, (dq, dk, dv, dth, dd) = _run(q, k, v, g, alpha, f, W, path)
    ro, rl, rq, rk, rv, rdd, rth = _reference(q, k, v, g, alpha, f, W)
    diff = np.abs(_f64(out) - ro)
    assert not (diff > bf16_out_tol(ro)).any(), f"out err {diff.max()}"
    assert float(np.max(np.abs(_f64(lse) - rl))) <= 1e-2
    for name, x, r in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv), ("dd", dd, rdd)):
        assert torch.isfinite(x.float()).all(), f"{name} not finite"
        e = _rel(_f64(x), r)
        assert e <= GRAD_TOL, f"{name} rel err {e}"
    eth = abs(float(dth[0]) - rth) / abs(rth)
    assert eth <= GRAD_TOL, f"dtheta {float(dth[0])} vs {rth} (rel {eth})"


SHAPES = [(1, 4, 4, 600, 8, 0.83), (2, 4, 2, 333, 6, 1.2173913)]


@pytest.mark.parametrize("path", ["mma", "residuals", "gather"])
@pytest.mark.parametrize("log2_scale", [-16, -20, -24])
@pytest.mark.parametrize("shape", SHAPES, ids=[f"B{s[0]}H{s[1]}kv{s[2]}T{s[3]}W{s[4]}" for s in SHAPES])
def test_small_upstream_gradients(shape, log2_scale, path):
    Bn, H, Hkv, T, W, alpha = shape
    f = fa.base("fib", 15)
    q, k, v = inputs.qkv(Bn, H, T, seed=T + 31, dtype=torch.bfloat16, Hkv=Hkv)
    g = (inputs.dout(Bn, H, T, seed=T + 32) * 2.0 ** log2_scale).to(torch.bfloat16)
    _check(q, k, v, g, alpha, f, W, path)


@pytest.mark.parametrize("path", ["mma", "residuals", "gather"])
def test_large_queries_small_keys(path):
    Bn, H, Hkv, T, W, alpha = SHAPES[0]
    f = fa.base("fib", 15)
    q, k, v = inputs.qkv(Bn, H, T, seed=T + 41, Hkv=Hkv)
    q = (q * 64.0).to(torch.bfloat16)
    k = (k / 64.0).to(torch.bfloat16)
    v = v.to(torch.bfloat16)
    g = inputs.dout(Bn, H, T, seed=T + 42, dtype=torch.bfloat16)
    _check(q, k, v, g, alpha, f, W, path)

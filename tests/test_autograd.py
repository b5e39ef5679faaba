"""The torch.autograd wrapper (Section 2: alpha = 0.5 + sigmoid(theta) is
trained through the attention).  CPU: the theta <-> alpha maps.  GPU: the
wrapper's gradients equal the C-ABI backward's, dtheta matches the oracle, and
a two-layer stack's theta gradients match finite differences of its loss."""
from __future__ import annotations

import math
import os

import numpy as np
import pytest
import torch

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs


def test_alpha_theta_maps():
    # both maps run in the library on fp32 host values: the round trip is
    # exact to fp32 rounding of alpha over the sigmoid's slope (at most ~5e-6
    # in theta at |theta| = 3)
    for th in (-3.0, -0.4, 0.0, 0.7, 2.5):
        a = fa.alpha_of_theta(th)
        assert 0.5 < a < 1.5
        assert abs(fa.theta_of_alpha(a) - th) < 3e-5
    assert fa.alpha_of_theta(0.0) == 1.0
    # the schedule of the library's learned kind is the same map
    th = [0.3, -1.2, 0.0]
    np.testing.assert_allclose(fa.alpha_schedule("learned", 3, theta=th), [fa.alpha_of_theta(t) for t in th],
                               rtol=0, atol=1e-6)


@pytest.mark.gpu
def test_wrapper_equals_abi_backward():
    q, k, v = inputs.qkv(2, 4, 300, seed=51, dtype=torch.bfloat16)
    g = inputs.dout(2, 4, 300, seed=52, dtype=torch.bfloat16).cuda()
    f = fa.base("fib", 15)
    theta = torch.tensor(0.37, device="cuda", requires_grad=True)
    qc, kc, vc = (t.cuda().requires_grad_(True) for t in (q, k, v))
    out = fa.fib_attention(qc, kc, vc, theta, f, 8)
    out.backward(g)
    alpha = fa.alpha_of_theta(0.37)
    # the wrapper (bf16) keeps the forward's rotated keys and residuals for its backward
    rk = fa.rotated_k_like(kc)
    res = fa.residuals_like(qc, 8, len(f))
    o2, l2 = fa.fwd(qc.detach(), kc.detach(), vc.detach(), alpha, f, 8, rotated_k=rk, residuals=res)
    dq, dk, dv, dth, _ = fa.bwd(qc.detach(), kc.detach(), vc.detach(), l2, g, alpha, f, 8, out=o2, rotated_k=rk,
                                residuals=res)
    torch.cuda.synchronize()
    assert torch.equal(out.detach(), o2)
    for a, b in ((qc.grad, dq), (kc.grad, dk), (vc.grad, dv)):
        assert torch.equal(a, b)
    assert float(theta.grad) == float(dth[0])


@pytest.mark.gpu
def test_wrapper_dtheta_against_oracle():
    q, k, v = inputs.qkv(1, 2, 200, seed=53, dtype=torch.float32)
    g = inputs.dout(1, 2, 200, seed=54, dtype=torch.float32)
    f = fa.base("fib", 15)
    theta = torch.tensor(-0.6, device="cuda", requires_grad=True)
    qc, kc, vc = (t.cuda() for t in (q, k, v))
    out = fa.fib_attention(qc, kc, vc, theta, f, 6)
    out.backward(g.cuda())
    a32 = float(np.float32(fa.alpha_of_theta(-0.6)))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    _, _, _, rdd = O.backward(q.double().numpy(), k.double().numpy(), v.double().numpy(), g.double().numpy(), 6, d)
    _, rth = O.dtheta(a32, f.astype(np.float64), rdd)
    assert abs(float(theta.grad) - rth) <= 1e-4 * max(1.0, abs(rth))


@pytest.mark.gpu
def test_stack_theta_gradients_match_finite_differences():
    """Two layers, q = k = v = the previous output (fp32): autograd's
    dL/dtheta_l against central differences of L = sum(out * g)."""
    torch.manual_seed(0)
    x = torch.randn(1, 2, 160, 64, device="cuda")
    gout = torch.randn(1, 2, 160, 64, device="cuda")
    f = fa.base("fib", 15)
    thetas = [0.45, -0.8]

    def loss(th):
        # fp64 sum: an fp32 sum of 20k terms carries ~1e-3 of rounding, as much
        # as a central difference with h = 1e-3 can resolve
        layers = [fa.FibAttention(W=4, offsets=f, theta=t, learned=True).cuda() for t in th]
        out = fa.attention_stack(x, layers)
        return (out.double() * gout.double()).sum(), layers

    L0, layers = loss(thetas)
    L0.backward()
    grads = [float(l.theta.grad) for l in layers]
    h = 1e-3                                     # moves no d_k across an integer at these thetas and T
    for i in range(2):
        tp = list(thetas); tp[i] += h
        tm = list(thetas); tm[i] -= h
        with torch.no_grad():
            fd = (float(loss(tp)[0]) - float(loss(tm)[0])) / (2 * h)
        assert abs(grads[i] - fd) <= 2e-3 * max(1.0, abs(fd)), (i, grads[i], fd)


@pytest.mark.gpu
def test_sixteen_layer_stack_runs_all_schedules():
    torch.manual_seed(1)
    x = torch.randn(2, 8, 1024, 64, device="cuda").to(torch.bfloat16).requires_grad_(True)
    f = fa.base("fib", 15)
    for kind in ("fixed", "linear", "coprime", "learned"):
        th = inputs.theta_learned(16, seed=3) if kind == "learned" else None
        alphas = fa.alpha_schedule(kind, 16, theta=th)
        layers = [fa.FibAttention(W=8, offsets=f, theta=fa.theta_of_alpha(float(a)), learned=(kind == "learned")).cuda()
                  for a in alphas]
        out = fa.attention_stack(x, layers)
        out.float().sum().backward()
        assert torch.isfinite(x.grad.float()).all()
        x.grad = None
        if kind == "learned":
            assert all(torch.isfinite(l.theta.grad) for l in layers)


@pytest.mark.gpu
def test_stack_reads_thetas_once_with_identical_results():
    """attention_stack passes each layer the host alpha it read for all layers
    in one copy; the result and the gradients equal those of layers that each
    read their own theta."""
    torch.manual_seed(2)
    x = torch.randn(1, 4, 300, 64, device="cuda").to(torch.bfloat16)
    gout = torch.randn_like(x)
    f = fa.base("fib", 15)
    thetas = [0.3, -1.1, 0.9]

    def run(stacked):
        xi = x.clone().requires_grad_(True)
        layers = [fa.FibAttention(W=8, offsets=f, theta=t, learned=True).cuda() for t in thetas]
        if stacked:
            out = fa.attention_stack(xi, layers)
        else:
            out = xi
            for layer in layers:
                out = layer(out, out, out)
        (out.float() * gout.float()).sum().backward()
        return out.detach(), xi.grad, [l.theta.grad.clone() for l in layers]

    o1, g1, t1 = run(True)
    o2, g2, t2 = run(False)
    assert torch.equal(o1, o2) and torch.equal(g1, g2)
    assert all(torch.equal(a, b) for a, b in zip(t1, t2))

"""torch.autograd wrapper of the C-ABI forward and backward.

The paper trains the per-layer scalar alpha = 0.5 + sigmoid(theta) together
with the model through this attention (arXiv 2606.28560, Section 2, "The
per-layer scalar" and "Implementation note").  `FibAttentionFunction` runs
`fibattn_fwd` and `fibattn_bwd`; the forward keeps the RoPE-rotated keys for
the backward (in place of k, the same size), so the backward does not rotate
k again, and with bf16 I/O also its residuals (the rotated queries, p of every
attended slot and the rung score differences), so the backward does not
recompute the scores.  alpha is a host value of the C ABI -- the kernels' shared-memory
layout depends on the rung distances -- so a theta held on the GPU is read
once per call (a device-to-host copy that waits for the queued work), unless
the caller passes alpha: `attention_stack` reads the thetas of all its layers
in one copy.
"""
from __future__ import annotations


import torch

from . import binding as B


def alpha_of_theta(theta: float) -> float:
    """alpha = 0.5 + sigmoid(theta) (Section 2, "The per-layer scalar"), as the
    library computes it (fibattn_alpha_schedule, learned kind)."""
    return float(B.alpha_schedule("learned", 1, theta=[float(theta)])[0])


class FibAttentionFunction(torch.autograd.Function):
    """out = attention(q, k, v) over the window and the scaled-Fibonacci rungs
    at alpha = 0.5 + sigmoid(theta).  Gradients flow to q, k, v and theta
    (a 0-dim tensor); offsets, W and the options are constants."""

    @staticmethod
    def forward(ctx, q, k, v, theta, offsets, W, rope_base, scale, dedup, alpha=None):
        if alpha is None:
            alpha = alpha_of_theta(float(theta))
        rk = B.rotated_k_like(k)
        kw = dict(rope_base=rope_base, scale=scale, dedup=dedup, rotated_k=rk)
        res = None
        if q.dtype == torch.bfloat16:
            # the tensor-core forward also keeps p, the rung score differences and
            # the rotated queries, so the backward does not recompute the scores
            res = B.residuals_like(q, W, len(offsets))
            try:
                out, lse = B.fwd(q, k, v, alpha, offsets, W, residuals=res, **kw)
            except B.FibattnError as e:
                if e.status != B.FIBATTN_ERR_UNSUPPORTED:
                    raise
                res = None
        if res is None:
            out, lse = B.fwd(q, k, v, alpha, offsets, W, **kw)
            res = torch.empty(0, dtype=torch.uint8, device=q.device)
        ctx.save_for_backward(q, k, v, out, lse, rk, res)
        ctx.args = (alpha, offsets, W, rope_base, scale, dedup, theta.dtype, theta.device)
        return out

    @staticmethod
    def backward(ctx, dout):
        q, k, v, out, lse, rk, res = ctx.saved_tensors
        alpha, offsets, W, rope_base, scale, dedup, tdtype, tdev = ctx.args
        dq, dk, dv, dth, _ = B.bwd(q, k, v, lse, dout.contiguous(), alpha, offsets, W, out=out,
                                   rope_base=rope_base, scale=scale, dedup=dedup, rotated_k=rk,
                                   residuals=res if res.numel() else None)
        dtheta = dth.reshape(()).to(device=tdev, dtype=tdtype)
        return dq, dk, dv, dtheta, None, None, None, None, None, None


def fib_attention(q, k, v, theta, offsets=None, W: int = 8, *, rope_base: float = 1e4, scale=None,
                  dedup: bool = True, alpha=None):
    """Functional form.  q [B,H,T,64]; k, v [B,Hkv,T,64] (bf16 or fp32, CUDA,
    contiguous); theta a 0-dim tensor (requires_grad for the learned
    schedule); offsets the base sequence (default: Fibonacci, K = 15).
    ``alpha``: the host value 0.5 + sigmoid(theta), when the caller has it
    (skips reading theta)."""
    if offsets is None:
        offsets = B.base("fib", 15)
    if not torch.is_tensor(theta):
        theta = torch.tensor(float(theta))
    return FibAttentionFunction.apply(q, k, v, theta, offsets, W, rope_base, scale, dedup,
                                      None if alpha is None else float(alpha))


class FibAttention(torch.nn.Module):
    """One layer's attention with its own scalar theta (learned unless
    `learned=False`; alpha = 0.5 + sigmoid(theta))."""

    def __init__(self, W: int = 8, offsets=None, theta: float = 0.0, learned: bool = True, rope_base: float = 1e4,
                 scale=None, dedup: bool = True):
        super().__init__()
        t = torch.tensor(float(theta))
        if learned:
            self.theta = torch.nn.Parameter(t)
        else:
            self.register_buffer("theta", t)
        self.W, self.rope_base, self.scale, self.dedup = W, rope_base, scale, dedup
        self.offsets = B.base("fib", 15) if offsets is None else offsets

    @property
    def alpha(self) -> float:
        return alpha_of_theta(float(self.theta))

    def forward(self, q, k, v, alpha=None):
        """``alpha``: the host value of 0.5 + sigmoid(theta), when the caller
        has read it (skips the per-call read of a theta on the GPU)."""
        return FibAttentionFunction.apply(q, k, v, self.theta, self.offsets, self.W, self.rope_base, self.scale,
                                          self.dedup, None if alpha is None else float(alpha))


def theta_of_alpha(alpha: float) -> float:
    """Inverse of alpha_of_theta on [0.5, 1.5] (fibattn_theta_of_alpha); the
    ends map to -/+ infinity, clamped to -/+ 30."""
    return float(B.theta_of_alpha_array([float(alpha)])[0])


def attention_stack(x: torch.Tensor, layers) -> torch.Tensor:
    """A stack of attention layers without projections: each layer attends
    with q = k = v = the previous layer's output (the first takes x).  The
    layers' thetas are read to the host in one copy before the first layer."""
    layers = list(layers)
    if not layers:
        return x
    dev = layers[0].theta.device
    thetas = torch.stack([layer.theta.detach().to(device=dev, dtype=torch.float32) for layer in layers]).tolist()
    alphas = B.alpha_schedule("learned", len(layers), theta=thetas)
    for layer, a in zip(layers, alphas):
        x = layer(x, x, x, alpha=float(a))
    return x

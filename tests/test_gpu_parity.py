"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs, element by element.

Tolerances: fp32 I/O max abs error <= 1e-4 on out/lse and <= 1e-4 relative
to the largest reference magnitude on gradients; bf16 I/O (fp32 accumulate)
max abs error <= 1e-2 on out and <= 3e-2 relative (max |g - ref| / max |ref|,
denominator floored at 1e-2) on gradients; dtheta |d - ref| / |ref|.
"""
from __future__ import annotations

import os

import numpy as np
import pytest
import torch

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs

pytestmark = pytest.mark.gpu

NTHREADS = max(1, min(16, os.cpu_count() or 1))
TOL = {torch.float32: dict(out=1e-4, lse=1e-4, grad=1e-4, dtheta=1e-4),
       torch.bfloat16: dict(out=1e-2, lse=1e-2, grad=3e-2, dtheta=3e-2)}


def _f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def bf16_out_tol(ref):
    """Per-element bar on bf16 outputs: 1e-2 wherever bf16 can hold it (|o| < 4,
    where half a bf16 ulp is at most 2^-8 * 2 = 2^-7).  For |o| >= 4 the format's
    own rounding step (half-ulp >= 2^-6) alone can exceed 1e-2 even for an exact
    result, so the excess of that half-ulp over 2^-7 is added to the bar."""
    e = np.floor(np.log2(np.maximum(np.abs(ref), 1e-30)))
    half_ulp = np.exp2(e - 8)
    return 1e-2 + np.maximum(0.0, half_ulp - 2.0 ** -7)


def _rel(a, ref):
    """max |a - ref| / max |ref|, the denominator floored at 1e-2.

    Some exact gradients are identically zero, e.g. dq of a query with a single
    attended slot, where softmax gives p = 1 and dq = scale p dp k (1 - p).  The
    kernel reaches that zero only up to the rounding of p = exp(s - lse) with
    lse stored in natural-log units: one ulp of p (6e-8) times scale |dp| |k|
    (about 3 at D = 64 with unit-normal inputs) leaves ~2e-7, so the floor must
    sit at least three decades above that for the fp32 bound of 1e-4."""
    return float(np.max(np.abs(a - ref)) / max(np.max(np.abs(ref)), 1e-2))


def _offsets(kind, K):
    return fa.base(kind, K)


def gpu_fwd(q, k, v, alpha, f, W, dedup=True, kernel="auto"):
    out, lse = fa.fwd(q.cuda(), k.cuda(), v.cuda(), alpha, f, W, dedup=dedup, kernel=kernel)
    torch.cuda.synchronize()
    return out, lse


def oracle_fwd(q, k, v, alpha, f, W, dedup=True):
    d = O.offsets_fp32(float(np.float32(alpha)), f.astype(np.float64))
    return O.forward(_f64(q), _f64(k), _f64(v), W, d, dedup=dedup, nthreads=NTHREADS)


def check_fwd(q, k, v, alpha, f, W, dedup=True, kernel="auto"):
    out, lse = gpu_fwd(q, k, v, alpha, f, W, dedup, kernel)
    ro, rl = oracle_fwd(q, k, v, alpha, f, W, dedup)
    tol = TOL[q.dtype]
    diff = np.abs(_f64(out) - ro)
    eo = float(np.max(diff)) if ro.size else 0.0
    el = float(np.max(np.abs(_f64(lse) - rl))) if rl.size else 0.0
    if q.dtype == torch.bfloat16 and ro.size:
        bad = diff > bf16_out_tol(ro)
        assert not bad.any(), f"out err {eo} (worst over bar at |ref|={np.abs(ro[bad]).max():.3f})"
        assert float(np.max(diff[np.abs(ro) < 4.0], initial=0.0)) <= tol["out"], f"out max abs err {eo} for |ref| < 4"
    else:
        assert eo <= tol["out"], f"out max abs err {eo}"
    assert el <= tol["lse"], f"lse max abs err {el}"
    return out, lse


def check_bwd(q, k, v, dout, alpha, f, W, dedup=True, kernel="auto"):
    """kernel: backward query pass ("gather" runs without the forward output)."""
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), dout.cuda()
    out, lse = fa.fwd(qc, kc, vc, alpha, f, W, dedup=dedup)
    dq, dk, dv, dth, dd = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, dedup=dedup, kernel=kernel,
                                 out=None if kernel == "gather" else out)
    torch.cuda.synchronize()
    a32 = float(np.float32(alpha))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    rq, rk, rv, rdd = O.backward(_f64(q), _f64(k), _f64(v), _f64(dout), W, d, dedup=dedup, nthreads=NTHREADS)
    _, rth = O.dtheta(a32, f.astype(np.float64), rdd)
    tol = TOL[q.dtype]
    for name, g, r in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv)):
        e = _rel(_f64(g), r)
        assert e <= tol["grad"], f"{name} rel err {e}"
    eth = abs(float(dth[0]) - rth) / max(abs(rth), 1e-6)
    assert eth <= tol["dtheta"], f"dtheta {float(dth[0])} vs {rth} (rel {eth})"
    edd = _rel(_f64(dd), rdd) if len(f) else 0.0
    assert edd <= tol["dtheta"], f"dd rel err {edd}"
    return dict(dq=dq, dk=dk, dv=dv, dtheta=float(dth[0]), dtheta_ref=rth)


# ------------------------------------------------------------ small cases --

SMALL = [
    # (B, H, Hkv, T, W, alpha, base, K, dedup)
    (1, 2, 2, 1, 8, 1.0, "fib", 15, True),
    (1, 2, 2, 5, 0, 1.0, "fib", 15, True),
    (2, 4, 2, 77, 3, 0.7333333, "fib", 15, True),
    (1, 3, 3, 130, 8, 1.0, "fib", 15, True),
    (2, 2, 1, 300, 12, 1.4666666, "fib", 15, True),
    (1, 2, 2, 257, 6, 0.5, "fib", 15, True),
    (1, 2, 2, 200, 10, 1.5, "fib", 15, True),
    (1, 2, 2, 190, 8, 0.9, "pow2", 10, True),
    (1, 2, 2, 150, 4, 1.1, "fib", 12, False),
    (1, 2, 2, 100, 5, 0.8, "fib", 0, True),
    (1, 2, 2, 64, 63, 1.0, "fib", 15, True),
    (1, 1, 1, 2100, 8, 1.5, "fib", 15, True),
    # slabs that start inside the 8-row rounding of the interval before them
    # (rung 11 at alpha 0.87, T 333; rung 11 at the alpha of a learned stack, T 1024)
    (2, 4, 2, 333, 8, 0.87, "fib", 15, True),
    (1, 2, 2, 1024, 8, 0.8801671, "fib", 15, True),
]


def _random_cases(n=16, seed=2606):
    """Seeded shapes across the launch paths: grouped-query heads (G = 1, 2, 4),
    lengths from 1 to 700 (ragged last tiles), W = 0..16, fractional alpha
    over [0.5, 1.5], both bases, K = 0..15, dedup on and off."""
    rng = np.random.default_rng(seed)
    cases = []
    for _ in range(n):
        Hkv = int(rng.integers(1, 3))
        G = int(rng.choice([1, 2, 4]))
        base = str(rng.choice(["fib", "pow2"]))
        K = int(rng.integers(0, 16 if base == "fib" else 11))
        cases.append((int(rng.integers(1, 3)), Hkv * G, Hkv, int(rng.integers(1, 701)), int(rng.integers(0, 17)),
                      float(np.float32(rng.uniform(0.5, 1.5))), base, K, bool(rng.integers(0, 2))))
    return cases


FWD_KERNELS = [(torch.float32, "auto"), (torch.bfloat16, "gather"), (torch.bfloat16, "mma")]


@pytest.mark.parametrize("dtype,kernel", FWD_KERNELS, ids=["f32", "bf16-gather", "bf16-mma"])
@pytest.mark.parametrize("case", SMALL, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in SMALL])
def test_forward_small(case, dtype, kernel):
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T + W, dtype=dtype, Hkv=Hkv)
    try:
        check_fwd(q, k, v, alpha, _offsets(base, K), W, dedup, kernel)
    except fa.FibattnError as e:
        if e.status == 2:                        # kernel does not apply to this shape
            pytest.skip(str(e))
        raise


BWD_KERNELS = [(torch.float32, "gather"), (torch.bfloat16, "gather"), (torch.bfloat16, "mma")]


@pytest.mark.parametrize("dtype,kernel", BWD_KERNELS, ids=["f32", "bf16-gather", "bf16-mma"])
@pytest.mark.parametrize("case", SMALL, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in SMALL])
def test_backward_small(case, dtype, kernel):
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T + W + 1, dtype=dtype, Hkv=Hkv)
    g = inputs.dout(Bn, H, T, seed=T + W + 2, dtype=dtype)
    try:
        check_bwd(q, k, v, g, alpha, _offsets(base, K), W, dedup, kernel)
    except fa.FibattnError as e:
        if e.status == 2:                        # kernel does not apply to this shape
            pytest.skip(str(e))
        raise


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32], ids=["bf16", "f32"])
def test_rotated_keys_from_the_forward(dtype):
    """The backward given the forward's rotated keys equals the backward that
    rotates k itself, bit for bit (same rotation, same kernels)."""
    q, k, v = inputs.qkv(2, 4, 333, seed=41, dtype=dtype, Hkv=2)
    g = inputs.dout(2, 4, 333, seed=42, dtype=dtype)
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), g.cuda()
    f = _offsets("fib", 15)
    rk = fa.binding.rotated_k_like(kc)
    out, lse = fa.fwd(qc, kc, vc, 0.9, f, 8, rotated_k=rk)
    out2, lse2 = fa.fwd(qc, kc, vc, 0.9, f, 8)
    r1 = fa.bwd(qc, kc, vc, lse, gc, 0.9, f, 8, out=out, rotated_k=rk)
    r2 = fa.bwd(qc, kc, vc, lse, gc, 0.9, f, 8, out=out)
    torch.cuda.synchronize()
    assert torch.equal(out, out2) and torch.equal(lse, lse2)
    for a, b in zip(r1, r2):
        assert torch.equal(a, b)


@pytest.mark.parametrize("kernel", ["mma", "gather"])
def test_backward_without_rung_gradients(kernel):
    """dtheta = dd = NULL (a fixed schedule): the same dq, dk, dv, bit for bit,
    without the rung-distance gradient."""
    q, k, v = inputs.qkv(2, 4, 260, seed=61, dtype=torch.bfloat16, Hkv=2)
    g = inputs.dout(2, 4, 260, seed=62, dtype=torch.bfloat16)
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), g.cuda()
    f = _offsets("fib", 15)
    for alpha in (1.0, 0.83):
        out, lse = fa.fwd(qc, kc, vc, alpha, f, 8)
        full = fa.bwd(qc, kc, vc, lse, gc, alpha, f, 8, out=out, kernel=kernel)
        lean = fa.bwd(qc, kc, vc, lse, gc, alpha, f, 8, out=out, kernel=kernel, rung_grads=False)
        torch.cuda.synchronize()
        assert lean[3] is None and lean[4] is None
        for a, b in zip(full[:3], lean[:3]):
            assert torch.equal(a, b)


def test_empty_batch():
    q = torch.zeros((0, 2, 16, 64), device="cuda")
    out, lse = fa.fwd(q, q, q, 1.0, _offsets("fib", 15), 4)
    assert out.shape == q.shape and lse.shape == (0, 2, 16)
    dq, dk, dv, dth, dd = fa.bwd(q, q, q, lse, q, 1.0, _offsets("fib", 15), 4)
    torch.cuda.synchronize()
    assert float(dth[0]) == 0.0 and torch.all(dd == 0)


def test_outputs_finite_and_deterministic():
    q, k, v = inputs.qkv(2, 4, 700, seed=5, dtype=torch.bfloat16)
    g = inputs.dout(2, 4, 700, seed=6, dtype=torch.bfloat16)
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), g.cuda()
    f = _offsets("fib", 15)
    for kernel in ("gather", "mma"):
        o1, l1 = fa.fwd(qc, kc, vc, 0.77, f, 8)
        r1 = fa.bwd(qc, kc, vc, l1, gc, 0.77, f, 8, out=o1, kernel=kernel)
        o2, l2 = fa.fwd(qc, kc, vc, 0.77, f, 8)
        r2 = fa.bwd(qc, kc, vc, l2, gc, 0.77, f, 8, out=o2, kernel=kernel)
        torch.cuda.synchronize()
        for a, b in zip(r1, r2):
            assert torch.equal(a, b)
            assert torch.isfinite(a.float()).all()


# --------------------------------------------- full-size workload configs --

def test_config1_fp32_alpha1_full():
    """B=1 H=8 T=1024 D=64 W=8 alpha=1 (integer rungs), fp32, seed 0: every output."""
    q, k, v = inputs.qkv(1, 8, 1024, seed=0, dtype=torch.float32)
    check_fwd(q, k, v, 1.0, _offsets("fib", 15), 8)


@pytest.mark.parametrize("W", [6, 8, 10, 12])
def test_config2_bf16_linear_stagger(W):
    """B=16 H=8 T=1024, 16 layers with alpha_l = 0.5 + l/15: layers 0, 7, 15 in
    full (all 131072 query heads of the launch)."""
    alphas = fa.alpha_schedule("linear", 16)
    f = _offsets("fib", 15)
    for layer in (0, 7, 15):
        q, k, v = inputs.qkv(16, 8, 1024, seed=inputs.layer_seed(1, layer), dtype=torch.bfloat16)
        check_fwd(q, k, v, float(alphas[layer]), f, W)


def test_config3_bf16_extrapolation_coprime():
    """B=4 H=8 T=4096 W=10, coprime-reassigned stagger: layers 0, 1, 9."""
    alphas = fa.alpha_schedule("coprime", 16)
    f = _offsets("fib", 15)
    for layer in (0, 1, 9):
        q, k, v = inputs.qkv(4, 8, 4096, seed=inputs.layer_seed(2, layer), dtype=torch.bfloat16)
        check_fwd(q, k, v, float(alphas[layer]), f, 10)


def test_config4_bf16_backward_learned_alpha():
    """B=16 H=8 T=1024 W=8, theta_l ~ N(0, 0.5): fwd+bwd of layers 0 and 15 in full."""
    theta = inputs.theta_learned(16, seed=3)
    alphas = fa.alpha_schedule("learned", 16, theta=theta)
    f = _offsets("fib", 15)
    for layer in (0, 15):
        s = inputs.layer_seed(3, layer)
        q, k, v = inputs.qkv(16, 8, 1024, seed=s, dtype=torch.bfloat16)
        g = inputs.dout(16, 8, 1024, seed=s, dtype=torch.bfloat16)
        check_bwd(q, k, v, g, float(alphas[layer]), f, 8, kernel="mma")
        if layer == 0:
            check_bwd(q, k, v, g, float(alphas[layer]), f, 8, kernel="gather")


def test_gqa_paper_shape_fwd_bwd():
    """The paper's head split (H = 8 query heads, Hkv = 2 kv heads: groups of
    4 sharing staged keys and values), B = 4, T = 1024, W = 8, learned alpha:
    forward and backward against the oracle in full."""
    theta = inputs.theta_learned(16, seed=3)
    alphas = fa.alpha_schedule("learned", 16, theta=theta)
    f = _offsets("fib", 15)
    for layer in (2, 11):
        s = inputs.layer_seed(5, layer)
        q, k, v = inputs.qkv(4, 8, 1024, seed=s, dtype=torch.bfloat16, Hkv=2)
        g = inputs.dout(4, 8, 1024, seed=s, dtype=torch.bfloat16)
        check_fwd(q, k, v, float(alphas[layer]), f, 8)
        check_bwd(q, k, v, g, float(alphas[layer]), f, 8, kernel="mma")


@pytest.mark.parametrize("base,K", [("fib", 15), ("pow2", 10)])
def test_config5_bf16_long_stress(base, K):
    """B=2 H=8 T=16384 W=12, linear stagger, Fibonacci vs power-of-2 base:
    fwd+bwd of layers 0, 7 (mid-ramp, alpha 0.9667) and 15 in full."""
    alphas = fa.alpha_schedule("linear", 16)
    f = _offsets(base, K)
    for layer in (0, 7, 15):
        s = inputs.layer_seed(4, layer)
        q, k, v = inputs.qkv(2, 8, 16384, seed=s, dtype=torch.bfloat16)
        g = inputs.dout(2, 8, 16384, seed=s, dtype=torch.bfloat16)
        check_fwd(q, k, v, float(alphas[layer]), f, 12)
        check_bwd(q, k, v, g, float(alphas[layer]), f, 12)


RANDOM = _random_cases(n=8, seed=1404)


@pytest.mark.parametrize("dtype,kernel", FWD_KERNELS, ids=["f32", "bf16-gather", "bf16-mma"])
@pytest.mark.parametrize("case", RANDOM, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]:.4f}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in RANDOM])
def test_forward_random_shapes(case, dtype, kernel):
    """Every forward kernel on seeded random shapes (see _random_cases)."""
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T * 17 + W, dtype=dtype, Hkv=Hkv)
    try:
        check_fwd(q, k, v, alpha, _offsets(base, K), W, dedup, kernel)
    except fa.FibattnError as e:
        if e.status == 2:
            pytest.skip(str(e))
        raise


@pytest.mark.parametrize("dtype,kernel", BWD_KERNELS, ids=["f32", "bf16-gather", "bf16-mma"])
@pytest.mark.parametrize("case", RANDOM, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]:.4f}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in RANDOM])
def test_backward_random_shapes(case, dtype, kernel):
    """Every backward query pass on seeded random shapes (see _random_cases)."""
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T * 17 + W + 1, dtype=dtype, Hkv=Hkv)
    g = inputs.dout(Bn, H, T, seed=T * 17 + W + 2, dtype=dtype)
    try:
        check_bwd(q, k, v, g, alpha, _offsets(base, K), W, dedup, kernel)
    except fa.FibattnError as e:
        if e.status == 2:
            pytest.skip(str(e))
        raise


# ------------------------------------------ rounded (integer) rung offsets --

def check_rounded(q, k, v, dout, alpha, f, W, kernel="auto", residuals=False):
    """The integer-offset variant (round_offsets): forward and backward (no
    rung gradient: the rounded distances do not vary with alpha) against the
    oracle on the rounded distances."""
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), dout.cuda()
    kw = dict(round_offsets=True)
    if residuals:
        kw.update(rotated_k=fa.rotated_k_like(kc), residuals=fa.residuals_like(qc, W, len(f)))
    out, lse = fa.fwd(qc, kc, vc, alpha, f, W, kernel="auto" if kernel != "gather" else "gather", **kw)
    dq, dk, dv, dth, dd = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, out=None if kernel == "gather" else out,
                                 kernel=kernel, rung_grads=False, **kw)
    torch.cuda.synchronize()
    d = O.offsets_rounded(float(np.float32(alpha)), f.astype(np.float64))
    ro, rl = O.forward(_f64(q), _f64(k), _f64(v), W, d, nthreads=NTHREADS)
    rq, rk, rv, _ = O.backward(_f64(q), _f64(k), _f64(v), _f64(dout), W, d, nthreads=NTHREADS)
    tol = TOL[q.dtype]
    diff = np.abs(_f64(out) - ro)
    if q.dtype == torch.bfloat16:
        assert not (diff > bf16_out_tol(ro)).any(), f"out err {diff.max()}"
    else:
        assert diff.max() <= tol["out"]
    assert float(np.max(np.abs(_f64(lse) - rl))) <= tol["lse"]
    for name, g, r in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv)):
        e = _rel(_f64(g), r)
        assert e <= tol["grad"], f"{name} rel err {e}"
    assert dth is None and dd is None


@pytest.mark.parametrize("kernel,dtype,residuals", [("mma", torch.bfloat16, False), ("mma", torch.bfloat16, True),
                                                    ("gather", torch.bfloat16, False),
                                                    ("gather", torch.float32, False)],
                         ids=["bf16-mma", "bf16-residuals", "bf16-gather", "f32"])
@pytest.mark.parametrize("kind,layer", [("linear", 5), ("linear", 12), ("coprime", 3)])
def test_rounded_stagger_small(kind, layer, kernel, dtype, residuals):
    alpha = float(fa.alpha_schedule(kind, 16)[layer])
    q, k, v = inputs.qkv(2, 4, 533, seed=layer + 90, dtype=dtype, Hkv=2)
    g = inputs.dout(2, 4, 533, seed=layer + 91, dtype=dtype)
    check_rounded(q, k, v, g, alpha, _offsets("fib", 15), 8, kernel, residuals)


def test_config2_rounded_linear_layer():
    """Config 2's shape (B=16 H=8 T=1024 W=8) at layer 7 of the linear stagger
    (alpha 0.9667) with the rung distances rounded: every output, and the
    training path's gradients."""
    alpha = float(fa.alpha_schedule("linear", 16)[7])
    s = inputs.layer_seed(1, 7)
    q, k, v = inputs.qkv(16, 8, 1024, seed=s, dtype=torch.bfloat16)
    g = inputs.dout(16, 8, 1024, seed=s, dtype=torch.bfloat16)
    check_rounded(q, k, v, g, alpha, _offsets("fib", 15), 8, "mma", residuals=True)

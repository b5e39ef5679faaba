"""GPU parity of the forward residuals (rotated queries, the unnormalised
softmax weight of every slot with 1 / (weight sum) per query, far-minus-floor
rung scores) and of the backward that reads them instead of recomputing the
scores.

Bars:
- out, lse of a forward that writes residuals: bit-identical to the forward
  without them (the same arithmetic; the residuals are extra stores).
- rotated q (bf16): |q~ - ref| <= 2^-8 |ref| + 1e-5 -- bf16 round-to-nearest
  (8 significant bits) of a value whose fp32 rotation is accurate to ~1e-6
  relative.
- p per slot, the stored weight times the stored 1 / (weight sum):
  |p - ref| <= 1e-2, the bf16 output bar (p is in [0, 1]; the scores come
  from fp16 operands); the row's p sum to 1 within 1e-2 (the forward's sum
  adds the bf16-rounded weights its value product uses, the stored weights
  are unrounded: a relative difference up to 2^-9).
- sd: |sd - ref| <= 2^-10 sum_e |q~_e| (|k~far_e| + |k~floor_e|) + 1e-4 --
  each fp16 factor carries at most 2^-11 relative rounding, accumulation fp32.
- gradients: the bf16 bars of the tensor-core backward against the oracle.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs
from tests.independent_forms import rope_complex_np
from tests.test_gpu_parity import NTHREADS, SMALL, TOL, _f64, _random_cases, _rel

pytestmark = pytest.mark.gpu


def _run_fwd(q, k, v, alpha, f, W, dedup):
    qc, kc, vc = q.cuda(), k.cuda(), v.cuda()
    res = fa.residuals_like(qc, W, len(f))
    res.fill_(0xAB)                              # every read entry must be written
    out_r, lse_r = fa.fwd(qc, kc, vc, alpha, f, W, dedup=dedup, residuals=res)
    out, lse = fa.fwd(qc, kc, vc, alpha, f, W, dedup=dedup)
    torch.cuda.synchronize()
    return res, out_r, lse_r, out, lse


@pytest.mark.parametrize("case", SMALL, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in SMALL])
def test_residuals_of_the_forward(case):
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T + W + 5, dtype=torch.bfloat16, Hkv=Hkv)
    f = fa.base(base, K)
    try:
        res, out_r, lse_r, out, lse = _run_fwd(q, k, v, alpha, f, W, dedup)
    except fa.FibattnError as e:
        if e.status == 2:                        # the tensor-core forward does not apply
            pytest.skip(str(e))
        raise
    assert torch.equal(out_r, out) and torch.equal(lse_r, lse)
    qt, P, sd, il = (x.cpu() for x in fa.residual_views(res, Bn, H, T, W, K))
    qf, kf = _f64(q), _f64(k)
    G = H // Hkv
    a32 = float(np.float32(alpha))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    p = fa.rung_params(np.float32(alpha), f, W, dedup=dedup)
    rng = np.random.default_rng(T + W)
    for b in range(Bn):
        for h in range(H):
            hk = h // G
            qr = rope_complex_np(qf[b, h])
            kr = rope_complex_np(kf[b, hk])
            got = qt[b, h].to(torch.float64).numpy()
            assert np.all(np.abs(got - qr) <= 2.0 ** -8 * np.abs(qr) + 1e-5)
            # every query up to 64 of them, the tail included
            idx = np.unique(np.concatenate([np.arange(min(T, 24)), np.arange(max(0, T - 24), T),
                                            rng.integers(0, T, size=16)]))
            for i in idx:
                sl = O.query_slots(qf[b, h], kf[b, hk], W, int(i), d, dedup=dedup)
                ref = np.zeros(W + 1 + K)
                for r0, r1, pr, rg in zip(sl["rows0"], sl["rows1"], sl["prob"], sl["rung"]):
                    ref[i - r0 if rg < 0 else W + 1 + rg] = pr
                    if rg >= 0:                  # far row r1 (row -1 reads zero), floor row r0
                        far = kr[r1] if r1 >= 0 else np.zeros(64)
                        sref = float(qr[i] @ (far - kr[r0]))
                        bound = 2.0 ** -10 * float(np.abs(qr[i]) @ (np.abs(far) + np.abs(kr[r0]))) + 1e-4
                        assert abs(float(sd[b, h, rg, i]) - sref) <= bound, (b, h, i, rg)
                # slots the key pass reads: window t = 0..W and every active rung
                want = np.zeros(W + 1 + K, dtype=bool)
                want[:W + 1] = True
                want[W + 1:] = p["active"] & (p["d"] <= T - 1)     # rungs within reach of the sequence
                gp = P[b, h, :, i].to(torch.float64).numpy() * float(il[b, h, i])
                assert np.all(np.abs(gp[want] - ref[want]) <= 1e-2), (b, h, i, gp[want], ref[want])
                # the weights of the attended slots sum to 1 / il (every attended slot is
                # stored, the others hold 0)
                assert abs(float(gp[want].sum()) - 1.0) <= 1e-2


def _check_bwd_residuals(q, k, v, dout, alpha, f, W, dedup=True, rung_grads=True):
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), dout.cuda()
    res = fa.residuals_like(qc, W, len(f))
    rk = fa.rotated_k_like(kc)
    out, lse = fa.fwd(qc, kc, vc, alpha, f, W, dedup=dedup, residuals=res, rotated_k=rk)
    dq, dk, dv, dth, dd = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, dedup=dedup, out=out, residuals=res,
                                 rotated_k=rk, kernel="mma", rung_grads=rung_grads)
    torch.cuda.synchronize()
    a32 = float(np.float32(alpha))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    rq, rkk, rv, rdd = O.backward(_f64(q), _f64(k), _f64(v), _f64(dout), W, d, dedup=dedup, nthreads=NTHREADS)
    tol = TOL[torch.bfloat16]
    for name, g, r in (("dq", dq, rq), ("dk", dk, rkk), ("dv", dv, rv)):
        e = _rel(_f64(g), r)
        assert e <= tol["grad"], f"{name} rel err {e}"
    if rung_grads:
        _, rth = O.dtheta(a32, f.astype(np.float64), rdd)
        eth = abs(float(dth[0]) - rth) / max(abs(rth), 1e-6)
        assert eth <= tol["dtheta"], f"dtheta {float(dth[0])} vs {rth} (rel {eth})"
        if len(f):
            assert _rel(_f64(dd), rdd) <= tol["dtheta"]
    else:
        assert dth is None and dd is None
    return dq, dk, dv


@pytest.mark.parametrize("case", SMALL, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in SMALL])
def test_backward_from_residuals(case):
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T + W + 7, dtype=torch.bfloat16, Hkv=Hkv)
    g = inputs.dout(Bn, H, T, seed=T + W + 8, dtype=torch.bfloat16)
    try:
        _check_bwd_residuals(q, k, v, g, alpha, fa.base(base, K), W, dedup)
    except fa.FibattnError as e:
        if e.status == 2:
            pytest.skip(str(e))
        raise


def test_backward_from_residuals_without_rung_gradients():
    """The fixed-schedule variant (no dtheta, no dd) gives the same dq, dk, dv
    bit for bit as the one with the rung gradient."""
    q, k, v = inputs.qkv(2, 4, 333, seed=71, dtype=torch.bfloat16, Hkv=2)
    g = inputs.dout(2, 4, 333, seed=72, dtype=torch.bfloat16)
    f = fa.base("fib", 15)
    full = _check_bwd_residuals(q, k, v, g, 0.87, f, 8)
    lean = _check_bwd_residuals(q, k, v, g, 0.87, f, 8, rung_grads=False)
    for a, b in zip(full, lean):
        assert torch.equal(a, b)


def test_backward_from_residuals_paper_shape():
    """B=2 H=8 Hkv=2 T=1024 W=8, learned-range alpha: the residual backward
    meets the oracle bar, and its gradients are within rounding (1e-2 relative)
    of the recomputing backward's."""
    Bn, H, Hkv, T, W, alpha = 2, 8, 2, 1024, 8, 1.2371
    q, k, v = inputs.qkv(Bn, H, T, seed=81, dtype=torch.bfloat16, Hkv=Hkv)
    g = inputs.dout(Bn, H, T, seed=82, dtype=torch.bfloat16)
    f = fa.base("fib", 15)
    dq, dk, dv = _check_bwd_residuals(q, k, v, g, alpha, f, W)
    qc, kc, vc, gc = q.cuda(), k.cuda(), v.cuda(), g.cuda()
    out, lse = fa.fwd(qc, kc, vc, alpha, f, W)
    dq2, dk2, dv2, _, _ = fa.bwd(qc, kc, vc, lse, gc, alpha, f, W, out=out, kernel="mma")
    torch.cuda.synchronize()
    for a, b in ((dq, dq2), (dk, dk2), (dv, dv2)):
        assert _rel(_f64(a), _f64(b)) <= 1e-2


def test_autograd_uses_residuals():
    """The autograd wrapper's gradients with residuals (bf16) meet the oracle bar."""
    Bn, H, T, W, alpha = 1, 2, 300, 8, 0.93
    q, k, v = inputs.qkv(Bn, H, T, seed=91, dtype=torch.bfloat16)
    g = inputs.dout(Bn, H, T, seed=92, dtype=torch.bfloat16)
    theta = torch.tensor(fa.theta_of_alpha(alpha), dtype=torch.float64, requires_grad=True)
    qc, kc, vc = (t.cuda().requires_grad_(True) for t in (q, k, v))
    out = fa.fib_attention(qc, kc, vc, theta, W=W)
    out.backward(g.cuda())
    torch.cuda.synchronize()
    a32 = float(np.float32(fa.alpha_of_theta(float(theta))))
    f = fa.base("fib", 15)
    d = O.offsets_fp32(a32, f.astype(np.float64))
    rq, rk, rv, rdd = O.backward(_f64(q), _f64(k), _f64(v), _f64(g), W, d, nthreads=NTHREADS)
    for name, a, r in (("dq", qc.grad, rq), ("dk", kc.grad, rk), ("dv", vc.grad, rv)):
        assert _rel(_f64(a), r) <= TOL[torch.bfloat16]["grad"], name
    _, rth = O.dtheta(a32, f.astype(np.float64), rdd)
    assert abs(float(theta.grad) - rth) / max(abs(rth), 1e-6) <= TOL[torch.bfloat16]["dtheta"]


def test_calls_from_a_fresh_host_thread():
    """A host thread that has made no CUDA call yet (a framework's backward
    worker) gets the same results as the main thread: the library binds the
    device's context before it encodes its tensor maps."""
    import threading
    q, k, v = (t.cuda() for t in inputs.qkv(1, 2, 300, seed=93, dtype=torch.bfloat16))
    g = inputs.dout(1, 2, 300, seed=94, dtype=torch.bfloat16).cuda()
    f = fa.base("fib", 15)
    res = fa.residuals_like(q, 8, 15)
    rk = fa.rotated_k_like(k)
    out, lse = fa.fwd(q, k, v, 0.93, f, 8, residuals=res, rotated_k=rk)
    main = {}
    for name, kw in (("res", dict(residuals=res, rotated_k=rk)), ("plain", {})):
        main[name] = fa.bwd(q, k, v, lse, g, 0.93, f, 8, out=out, **kw)
    got, err = {}, []

    def work():
        try:
            for name, kw in (("res", dict(residuals=res, rotated_k=rk)), ("plain", {})):
                got[name] = fa.bwd(q, k, v, lse, g, 0.93, f, 8, out=out, **kw)
            got["fwd"] = fa.fwd(q, k, v, 0.93, f, 8)
            torch.cuda.synchronize()
        except Exception as e:                    # surfaced in the main thread below
            err.append(e)
    th = threading.Thread(target=work)
    th.start()
    th.join()
    torch.cuda.synchronize()
    assert not err, err
    for name in ("res", "plain"):
        for a, b in zip(main[name][:3], got[name][:3]):
            assert torch.equal(a, b)
    assert torch.equal(got["fwd"][0], out)


RANDOM = _random_cases()


@pytest.mark.parametrize("case", RANDOM, ids=[f"B{c[0]}H{c[1]}kv{c[2]}T{c[3]}W{c[4]}a{c[5]:.4f}{c[6]}{c[7]}d{int(c[8])}"
                                              for c in RANDOM])
def test_random_shapes_forward_and_backward_from_residuals(case):
    """The residual forward's output and the backward from its residuals
    against the oracle on seeded random shapes."""
    from tests.test_gpu_parity import bf16_out_tol
    Bn, H, Hkv, T, W, alpha, base, K, dedup = case
    q, k, v = inputs.qkv(Bn, H, T, seed=T * 31 + W, dtype=torch.bfloat16, Hkv=Hkv)
    g = inputs.dout(Bn, H, T, seed=T * 31 + W + 1, dtype=torch.bfloat16)
    f = fa.base(base, K)
    try:
        res = fa.residuals_like(q.cuda(), W, K)
        out, _ = fa.fwd(q.cuda(), k.cuda(), v.cuda(), alpha, f, W, dedup=dedup, residuals=res)
    except fa.FibattnError as e:
        if e.status == 2:
            pytest.skip(str(e))
        raise
    torch.cuda.synchronize()
    d = O.offsets_fp32(float(np.float32(alpha)), f.astype(np.float64))
    ro, _ = O.forward(_f64(q), _f64(k), _f64(v), W, d, dedup=dedup, nthreads=NTHREADS)
    assert not (np.abs(_f64(out) - ro) > bf16_out_tol(ro)).any()
    _check_bwd_residuals(q, k, v, g, alpha, f, W, dedup)


@pytest.mark.parametrize("base,K", [("fib", 15), ("pow2", 10)])
def test_config5_training_path_mid_layer(base, K):
    """Config 5 (B=2 H=8 T=16384 W=12, linear stagger) through the path the
    long-sequence benchmark times -- the forward keeps its rotated keys and
    residuals, the backward reads them -- at the mid-ramp layer 7 (alpha
    0.9667), every gradient and dtheta against the oracle."""
    alpha = float(fa.alpha_schedule("linear", 16)[7])
    s = inputs.layer_seed(4, 7)
    q, k, v = inputs.qkv(2, 8, 16384, seed=s, dtype=torch.bfloat16)
    g = inputs.dout(2, 8, 16384, seed=s, dtype=torch.bfloat16)
    _check_bwd_residuals(q, k, v, g, alpha, fa.base(base, K), 12)


def test_gqa_training_path_bench_shape():
    """The grouped-query step the benchmark times (B=16 H=8 Hkv=2 T=1024 W=8,
    learned theta seed 3; the key pass takes one block per pass there, its
    grid being under two waves) through the residual path, layer 7, against
    the oracle."""
    theta = inputs.theta_learned(16, seed=3)
    alpha = float(fa.alpha_schedule("learned", 16, theta=theta)[7])
    s = inputs.layer_seed(3, 7)
    q, k, v = inputs.qkv(16, 8, 1024, seed=s, dtype=torch.bfloat16, Hkv=2)
    g = inputs.dout(16, 8, 1024, seed=s, dtype=torch.bfloat16)
    _check_bwd_residuals(q, k, v, g, alpha, fa.base("fib", 15), 8)


@pytest.mark.parametrize("layer", [0, 7, 12, 15])
def test_config4_training_path_full(layer):
    """Config 4 (B=16 H=8 T=1024 W=8, learned theta seed 3) through the path the
    benchmark times: the forward keeps its rotated keys and residuals, the
    backward reads them.  Every output and gradient of the layer against the
    oracle; layer 12 (alpha 0.8801671) is the layer whose staged slab once sat
    in the rounding padding of the interval before it."""
    theta = inputs.theta_learned(16, seed=3)
    alpha = float(fa.alpha_schedule("learned", 16, theta=theta)[layer])
    s = inputs.layer_seed(3, layer)
    q, k, v = inputs.qkv(16, 8, 1024, seed=s, dtype=torch.bfloat16)
    g = inputs.dout(16, 8, 1024, seed=s, dtype=torch.bfloat16)
    f = fa.base("fib", 15)
    qc, kc, vc = q.cuda(), k.cuda(), v.cuda()
    res = fa.residuals_like(qc, 8, 15)
    rk = fa.rotated_k_like(kc)
    out, lse = fa.fwd(qc, kc, vc, alpha, f, 8, residuals=res, rotated_k=rk)
    torch.cuda.synchronize()
    a32 = float(np.float32(alpha))
    d = O.offsets_fp32(a32, f.astype(np.float64))
    ro, rl = O.forward(_f64(q), _f64(k), _f64(v), 8, d, nthreads=NTHREADS)
    diff = np.abs(_f64(out) - ro)
    from tests.test_gpu_parity import bf16_out_tol
    assert not (diff > bf16_out_tol(ro)).any(), f"out err {diff.max()}"
    assert float(np.max(np.abs(_f64(lse) - rl))) <= 1e-2
    _check_bwd_residuals(q, k, v, g, alpha, f, 8)

"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Every check compares the oracle with something other than itself: an
independent dense boolean-mask attention, PyTorch's scaled_dot_product_attention
in its special cases, an interpolation-matrix formulation differentiated by
torch.autograd, finite differences, printed constants, and invariants.
"""
from __future__ import annotations

import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from tests.independent_forms import (bool_mask, masked_attention_np, matrix_attention_torch,
                                     rope_complex_torch)

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLD, name)) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            parts = line.split()
            if parts[0].replace(".", "").isdigit():
                vals.setdefault("_rows", []).append([float(x) for x in parts])
            else:
                vals[parts[0]] = [float(x) for x in parts[1:]]
    return vals


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


# --------------------------------------------------------------- bases ----

def test_fib_base_matches_paper():
    gold = _read_golden("fib_base.txt")["_rows"][0]
    np.testing.assert_array_equal(O.fib_base(15), gold)
    assert O.fib_base(15)[-1] == 987


def test_pow2_base():
    gold = _read_golden("pow2_base.txt")["_rows"][0]
    np.testing.assert_array_equal(O.pow2_base(10), gold)


def test_schedules_match_paper():
    g = _read_golden("schedules.txt")
    lin = O.alpha_schedule("linear", 16)
    assert lin[0] == g["linear_first"][0] and lin[-1] == g["linear_last"][0]
    np.testing.assert_allclose(np.diff(lin), 1.0 / 15, rtol=0, atol=1e-15)
    cop = O.alpha_schedule("coprime", 16, stride=int(g["coprime_stride"][0]))
    idx = [int(x) for x in g["coprime_index"]]
    np.testing.assert_array_equal(cop, lin[idx])
    # same multiset as the linear ramp; 7 is its own inverse mod 16 so the
    # two ways of reading the reassignment give one permutation
    np.testing.assert_array_equal(np.sort(cop), np.sort(lin))
    assert sorted(idx) == list(range(16))
    assert all((7 * idx[l]) % 16 == l for l in range(16))
    assert O.alpha_schedule("fixed", 16).tolist() == [1.0] * 16
    al = O.alpha_schedule("learned", 3, theta=[0.0, -50.0, 50.0])
    np.testing.assert_allclose(al, [g["learned_alpha_at_theta0"][0], g["alpha_min"][0], g["alpha_max"][0]], atol=1e-12)


def test_offsets_fp32_rounding():
    f = O.fib_base(15)
    d = O.offsets_fp32(1.0, f)
    np.testing.assert_array_equal(d, f)                     # alpha = 1: integer rungs
    a = 0.5 + 7 / 15
    d = O.offsets_fp32(a, f)
    expect = (np.float32(a) * f.astype(np.float32)).astype(np.float64)
    np.testing.assert_array_equal(d, expect)


# ----------------------------------------- integer alpha: bool-mask form --

@pytest.mark.parametrize("T,W,H,Hkv,seed", [(16, 3, 2, 2, 0), (64, 8, 4, 2, 1), (200, 0, 2, 1, 2),
                                            (130, 12, 2, 2, 3)])
def test_integer_alpha_equals_boolean_mask_attention(T, W, H, Hkv, seed):
    """At alpha = 1 every rung is an integer row: the interpolated gather is an
    exact gather and equals dense attention with a boolean mask (Section 2,
    "Implementation note": numerically identical)."""
    D = 16
    q, k, v = _rand((2, H, T, D), seed), _rand((2, Hkv, T, D), seed + 10), _rand((2, Hkv, T, D), seed + 20)
    f = O.fib_base(15)
    d = O.offsets_fp32(1.0, f)
    o, lse = O.forward(q, k, v, W, d)
    mask = bool_mask(T, W, f)
    o2, lse2 = masked_attention_np(q, k, v, mask, 1 / math.sqrt(D), kv_group=H // Hkv)
    np.testing.assert_allclose(o, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse2, rtol=0, atol=1e-12)


def test_integer_pow2_base_equals_boolean_mask():
    T, W, D = 100, 2, 8
    q, k, v = _rand((1, 2, T, D), 5), _rand((1, 2, T, D), 6), _rand((1, 2, T, D), 7)
    f = O.pow2_base(10)
    o, _ = O.forward(q, k, v, W, O.offsets_fp32(1.0, f))
    o2, _ = masked_attention_np(q, k, v, bool_mask(T, W, f), 1 / math.sqrt(D))
    np.testing.assert_allclose(o, o2, rtol=0, atol=1e-12)


def test_no_dedup_counts_duplicate_rungs_twice():
    """Reading check: without dedup a rung at d_k <= W is a second slot on the
    same row, i.e. that key gets weight 2 inside the softmax."""
    T, W, D = 40, 8, 8
    q, k, v = _rand((1, 1, T, D), 8), _rand((1, 1, T, D), 9), _rand((1, 1, T, D), 10)
    f = np.array([3.0])
    o, lse = O.forward(q, k, v, W, f, dedup=False)
    qt = rope_complex_torch(torch.tensor(q)).numpy()[0, 0]
    kt = rope_complex_torch(torch.tensor(k)).numpy()[0, 0]
    i = 20
    js = list(range(i - W, i + 1)) + [i - 3]
    s = np.array([qt[i] @ kt[j] for j in js]) / math.sqrt(D)
    p = np.exp(s - s.max()); p /= p.sum()
    expect = sum(pi * v[0, 0, j] for pi, j in zip(p, js))
    np.testing.assert_allclose(o[0, 0, i], expect, atol=1e-12)


# --------------------------------------------------- special cases -------

def test_dense_window_is_causal_attention():
    """W >= T-1 (dedup drops every rung inside the window, the rest reach before
    position 0): plain causal softmax attention, checked with PyTorch SDPA."""
    T, D, H = 48, 16, 3
    q, k, v = _rand((2, H, T, D), 11), _rand((2, H, T, D), 12), _rand((2, H, T, D), 13)
    o, lse = O.forward(q, k, v, T - 1, O.fib_base(15))
    qt = rope_complex_torch(torch.tensor(q))
    kt = rope_complex_torch(torch.tensor(k))
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, torch.tensor(v), is_causal=True)
    np.testing.assert_allclose(o, ref.numpy(), rtol=0, atol=1e-12)


def test_no_rungs_is_sliding_window_attention():
    T, D, W = 64, 16, 5
    q, k, v = _rand((1, 2, T, D), 14), _rand((1, 2, T, D), 15), _rand((1, 2, T, D), 16)
    o, _ = O.forward(q, k, v, W, np.zeros(0))
    i = torch.arange(T)[:, None]
    j = torch.arange(T)[None, :]
    mask = (i - j >= 0) & (i - j <= W)
    qt = rope_complex_torch(torch.tensor(q))
    kt = rope_complex_torch(torch.tensor(k))
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, torch.tensor(v), attn_mask=mask)
    np.testing.assert_allclose(o, ref.numpy(), rtol=0, atol=1e-12)


def test_single_position_and_empty_batch():
    q, k, v = _rand((1, 1, 1, 8), 17), _rand((1, 1, 1, 8), 18), _rand((1, 1, 1, 8), 19)
    o, lse = O.forward(q, k, v, 4, O.fib_base(15))
    np.testing.assert_allclose(o[0, 0, 0], v[0, 0, 0], atol=1e-15)     # self only
    qt = rope_complex_torch(torch.tensor(q)).numpy()[0, 0, 0]
    kt = rope_complex_torch(torch.tensor(k)).numpy()[0, 0, 0]
    np.testing.assert_allclose(lse[0, 0, 0], qt @ kt / math.sqrt(8), atol=1e-14)
    o, lse = O.forward(np.zeros((0, 2, 5, 8)), np.zeros((0, 2, 5, 8)), np.zeros((0, 2, 5, 8)), 2, O.fib_base(3))
    assert o.shape == (0, 2, 5, 8) and lse.shape == (0, 2, 5)


# -------------------------------------- fractional alpha: matrix form -----

DYADIC_ALPHAS = [0.5, 0.625, 0.8125, 1.1875, 1.375, 1.5]    # alpha * f_k exact in fp32


@pytest.mark.parametrize("alpha", DYADIC_ALPHAS)
def test_fractional_alpha_equals_interpolation_matrix(alpha):
    T, D, W, H, Hkv = 70, 8, 4, 4, 2
    f = O.fib_base(11)
    d = O.offsets_fp32(alpha, f)
    np.testing.assert_array_equal(d, alpha * f)     # dyadic: no fp32 rounding
    q, k, v = _rand((1, H, T, D), 20), _rand((1, Hkv, T, D), 21), _rand((1, Hkv, T, D), 22)
    o, lse = O.forward(q, k, v, W, d)
    o2, lse2 = matrix_attention_torch(torch.tensor(q), torch.tensor(k), torch.tensor(v), W,
                                      torch.tensor(d), 1 / math.sqrt(D), kv_group=H // Hkv)
    np.testing.assert_allclose(o, o2.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse2.numpy(), rtol=0, atol=1e-12)


@pytest.mark.parametrize("alpha,dedup", [(0.8125, True), (1.0, True), (1.375, False), (0.5, True)])
def test_backward_equals_autograd_of_matrix_form(alpha, dedup):
    T, D, W, H, Hkv = 48, 8, 3, 4, 2
    f = O.fib_base(9)
    q, k, v = _rand((2, H, T, D), 30), _rand((2, Hkv, T, D), 31), _rand((2, Hkv, T, D), 32)
    g = _rand((2, H, T, D), 33)
    d = O.offsets_fp32(alpha, f)
    dq, dk, dv, dd = O.backward(q, k, v, g, W, d, dedup=dedup)
    da, _ = O.dtheta(alpha, f, dd)

    qt, kt, vt = (torch.tensor(x, requires_grad=True) for x in (q, k, v))
    a = torch.tensor(alpha, dtype=torch.float64, requires_grad=True)
    dist = a * torch.tensor(f)
    o, _ = matrix_attention_torch(qt, kt, vt, W, dist, 1 / math.sqrt(D), dedup=dedup, kv_group=H // Hkv)
    (o * torch.tensor(g)).sum().backward()
    np.testing.assert_allclose(dq, qt.grad.numpy(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(dk, kt.grad.numpy(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(dv, vt.grad.numpy(), rtol=0, atol=1e-11)
    np.testing.assert_allclose(da, a.grad.item(), rtol=1e-10, atol=1e-10)


# ------------------------------------------------- finite differences ----

def _loss(q, k, v, g, W, d):
    o, _ = O.forward(q, k, v, W, d)
    return float((o * g).sum())


def _safe_theta(f, W, T, h):
    """A theta whose rung distances sit well away from integers, from W and
    from every position, so +-h does not cross a floor or a mask boundary."""
    for theta in np.linspace(-1.3, 1.3, 261):
        a = 0.5 + 1 / (1 + math.exp(-theta))
        d = a * f
        margin = f * 0.25 * h * 4
        frac = d - np.floor(d)
        if np.all(np.minimum(frac, 1 - frac) > margin + 1e-3) and np.all(np.abs(d - W) > 1e-3):
            return theta
    raise RuntimeError("no safe theta")


def test_dtheta_matches_finite_difference():
    T, D, W, H = 60, 8, 3, 2
    f = O.fib_base(10)
    h = 1e-6
    theta = _safe_theta(f, W, T, h)
    q, k, v, g = (_rand((1, H, T, D), s) for s in (40, 41, 42, 43))

    def d_of(t):
        return (0.5 + 1 / (1 + math.exp(-t))) * f               # fp64 distances

    alpha = 0.5 + 1 / (1 + math.exp(-theta))
    _, _, _, dd = O.backward(q, k, v, g, W, d_of(theta))
    _, dth = O.dtheta(alpha, f, dd)
    fd = (_loss(q, k, v, g, W, d_of(theta + h)) - _loss(q, k, v, g, W, d_of(theta - h))) / (2 * h)
    assert abs(dth) > 1e-3
    np.testing.assert_allclose(dth, fd, rtol=2e-6, atol=1e-8)
    # per-rung distance derivatives
    for kk in range(len(f)):
        dp = d_of(theta).copy(); dm = dp.copy()
        dp[kk] += h; dm[kk] -= h
        fdk = (_loss(q, k, v, g, W, dp) - _loss(q, k, v, g, W, dm)) / (2 * h)
        np.testing.assert_allclose(dd[kk], fdk, rtol=1e-5, atol=1e-7)


def test_dqkv_match_finite_difference():
    T, D, W, H, Hkv = 40, 8, 2, 2, 1
    f = O.fib_base(9)
    d = O.offsets_fp32(0.8125, f)
    q, k, v, g = _rand((1, H, T, D), 50), _rand((1, Hkv, T, D), 51), _rand((1, Hkv, T, D), 52), _rand((1, H, T, D), 53)
    dq, dk, dv, _ = O.backward(q, k, v, g, W, d)
    rng = np.random.default_rng(54)
    h = 1e-6
    for name, x, gx in (("q", q, dq), ("k", k, dk), ("v", v, dv)):
        for _ in range(6):
            idx = tuple(int(rng.integers(0, s)) for s in x.shape)
            xp = x.copy(); xp[idx] += h
            xm = x.copy(); xm[idx] -= h
            args = {"q": q, "k": k, "v": v}
            lp = _loss(*(xp if n == name else args[n] for n in "qkv"), g, W, d)
            lm = _loss(*(xm if n == name else args[n] for n in "qkv"), g, W, d)
            np.testing.assert_allclose(gx[idx], (lp - lm) / (2 * h), rtol=1e-6, atol=1e-8)


def test_dtheta_nonzero_at_integer_alpha_one_sided():
    """Section 2: interpolation keeps a nonzero alpha-gradient even when every
    rung sits on an integer position.  The floor-of-distance reading makes it
    the one-sided derivative from above; check against a forward difference."""
    T, D, W = 80, 8, 4
    f = O.fib_base(10)
    q, k, v, g = (_rand((1, 2, T, D), s) for s in (60, 61, 62, 63))
    # a rung with d_k == i sits on the mask boundary d_k > i: moving d up masks
    # it (a jump, not a derivative).  Give those queries no upstream gradient.
    g[..., [int(x) for x in f if x < T], :] = 0.0
    d = O.offsets_fp32(1.0, f)
    _, _, _, dd = O.backward(q, k, v, g, W, d)
    da, dth = O.dtheta(1.0, f, dd)
    assert abs(dth) > 1e-4 and dth == pytest.approx(da * 0.25)
    h = 1e-7
    fd = (_loss(q, k, v, g, W, (1.0 + h) * f) - _loss(q, k, v, g, W, f)) / h
    np.testing.assert_allclose(da, fd, rtol=2e-5, atol=1e-6)


# ------------------------------------------------------- invariants -------

@pytest.mark.parametrize("alpha", [1.0, 0.7333333, 1.4666666])
def test_slot_invariants(alpha):
    T, D, W = 300, 8, 6
    f = O.fib_base(15)
    d = O.offsets_fp32(alpha, f)
    q, k = _rand((T, D), 70), _rand((T, D), 71)
    for i in [0, 1, 5, 6, 7, 20, 143, 144, 233, 299]:
        s = O.query_slots(q, k, W, i, d)
        assert abs(s["prob"].sum() - 1.0) < 1e-14
        # self position is always present with positive probability
        self_slot = np.where((s["rows0"] == i) & (s["rung"] == -1))[0]
        assert len(self_slot) == 1 and s["prob"][self_slot[0]] > 0
        # window rows
        win = s["rows0"][s["rung"] == -1]
        assert sorted(win.tolist()) == list(range(max(0, i - W), i + 1))
        # rungs: only those with W < d_k <= i appear; rows and weights follow
        rk = s["rung"][s["rung"] >= 0]
        expect = [kk for kk in range(len(f)) if W < d[kk] <= i]
        assert rk.tolist() == expect
        for j in np.where(s["rung"] >= 0)[0]:
            kk = s["rung"][j]
            s0 = math.floor(d[kk]); w = d[kk] - s0
            assert s["rows0"][j] == i - s0 and s["rows1"][j] == i - s0 - 1
            assert s["c0"][j] == pytest.approx(1 - w, abs=1e-15) and s["c1"][j] == pytest.approx(w, abs=1e-15)
            assert s["rows1"][j] >= 0 or s["c1"][j] == 0.0


def test_masked_rung_rows_do_not_leak():
    """A rung reaching before position 0 is masked: perturbing key/value rows
    that only such a rung could read leaves the output unchanged."""
    T, D, W = 120, 8, 2
    f = np.array([50.0, 100.0])
    q, k, v = _rand((1, 1, T, D), 80), _rand((1, 1, T, D), 81), _rand((1, 1, T, D), 82)
    o, _ = O.forward(q, k, v, W, f)
    # query 60: rung 100 masked (100 > 60); rung 50 reads row 10.  Rows 0..9 are
    # read by query 60 only through the masked rung -> perturb them.
    k2, v2 = k.copy(), v.copy()
    k2[0, 0, :10] += 5.0; v2[0, 0, :10] -= 3.0
    o2, _ = O.forward(q, k2, v2, W, f)
    np.testing.assert_array_equal(o[0, 0, 60:62], o2[0, 0, 60:62])
    assert not np.allclose(o[0, 0, 100:110], o2[0, 0, 100:110])


def test_rung_exactly_at_position_reads_row_zero():
    T, D, W = 30, 4, 1
    f = np.array([13.0])
    q, k = _rand((T, D), 90), _rand((T, D), 91)
    s = O.query_slots(q, k, W, 13, f)
    j = np.where(s["rung"] == 0)[0]
    assert len(j) == 1 and s["rows0"][j[0]] == 0 and s["rows1"][j[0]] == -1 and s["c1"][j[0]] == 0.0
    s = O.query_slots(q, k, W, 12, f)
    assert (s["rung"] == 0).sum() == 0


def test_rope_relative_position_invariance():
    """RoPE at true positions makes a score depend on i-j only: with every q
    row equal and every k row equal, all queries with a full slot set see the
    same scores, hence the same lse."""
    T, D, W = 200, 16, 3
    f = np.array([5.0, 9.5, 31.25])
    rng = np.random.default_rng(100)
    q = np.broadcast_to(rng.standard_normal(D), (1, 1, T, D)).copy()
    k = np.broadcast_to(rng.standard_normal(D), (1, 1, T, D)).copy()
    v = rng.standard_normal((1, 1, T, D))
    _, lse = O.forward(q, k, v, W, f)
    full = lse[0, 0, 33:]
    np.testing.assert_allclose(full, full[0], rtol=0, atol=1e-12)
    assert np.ptp(lse[0, 0, :33]) > 1e-6     # partial slot sets differ


def test_oracle_threads_agree():
    T, D, W = 64, 8, 3
    q, k, v, g = (_rand((2, 4, T, D), s) for s in (110, 111, 112, 113))
    d = O.offsets_fp32(0.9, O.fib_base(10))
    a = O.forward(q, k, v, W, d, nthreads=1)
    b = O.forward(q, k, v, W, d, nthreads=4)
    np.testing.assert_array_equal(a[0], b[0])
    ga = O.backward(q, k, v, g, W, d, nthreads=1)
    gb = O.backward(q, k, v, g, W, d, nthreads=4)
    for x, y in zip(ga, gb):
        np.testing.assert_array_equal(x, y)


# ---------------------------------- rounded offsets: the boolean-mask path --

def _rounded_independently(alpha, f):
    """Integer distances by another route than the oracle's: Python's round()
    (ties to even) of the fp32 product."""
    return [round(float(np.float32(np.float32(alpha) * np.float32(x)))) for x in f]


def test_rounded_offsets_ties_to_even():
    f = O.fib_base(15)
    # alpha 0.5: 0.5 -> 0, 1.5 -> 2, 2.5 -> 2, 6.5 -> 6, 10.5 -> 10, 27.5 -> 28, 44.5 -> 44
    d = O.offsets_rounded(0.5, f)
    assert list(d[:11]) == [0, 1, 2, 2, 4, 6, 10, 17, 28, 44, 72]
    for alpha in (0.5, 0.7333333, 1.0, 1.1, 1.5):
        assert list(O.offsets_rounded(alpha, f)) == _rounded_independently(alpha, f)


@pytest.mark.parametrize("kind,layers", [("linear", (1, 5, 11, 14)), ("coprime", (1, 3, 9))])
@pytest.mark.parametrize("T,W", [(64, 8), (200, 6), (300, 12)])
def test_rounded_stagger_equals_boolean_mask_attention(kind, layers, T, W):
    """The rounded linear and coprime staggers are integer gathers: the oracle
    on the rounded distances equals dense attention with the boolean mask of
    those integer distances (Section 2, "Implementation note": numerically
    identical), in dedup mode (the attended set is a union)."""
    D = 16
    f = O.fib_base(15)
    alphas = O.alpha_schedule(kind, 16)
    for l in layers:
        q, k, v = _rand((1, 2, T, D), 100 + l), _rand((1, 2, T, D), 200 + l), _rand((1, 2, T, D), 300 + l)
        d = O.offsets_rounded(float(alphas[l]), f)
        o, lse = O.forward(q, k, v, W, d)
        o2, lse2 = masked_attention_np(q, k, v, bool_mask(T, W, _rounded_independently(float(alphas[l]), f)),
                                       1 / math.sqrt(D))
        np.testing.assert_allclose(o, o2, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, lse2, rtol=0, atol=1e-12)

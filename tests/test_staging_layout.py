"""The shared-memory staging layout of the tensor-core kernels, checked on the
CPU through the C ABI: every staged slab (and the window band) must map to
consecutive shared rows holding consecutive sequence rows.

A tile of 120 queries (keys) reads, per rung, a slab of 122 (121) rows; the library
merges overlapping row ranges and rounds each merged interval up to whole
8-row copies.  An earlier merge rule compared the next range with the
previous one's unrounded end, so a slab starting inside the rounding padding
of the interval before it was mapped into that padding (three rows off for
alpha = 0.87, T = 333, rung 11); these cases pin the rule that rounded
intervals never overlap.
"""
from __future__ import annotations

import numpy as np
import pytest

import paper_2606_28560_gb300 as fa

M1 = 121                                          # a tile of 120 rows plus one


def _ranges(kind, W, s0s):
    Wp = 0 if W == 0 else (8 if W <= 8 else 16)
    if kind == "query":
        return [(-Wp, M1)], [(-s - 1, M1 - s) for s in s0s]
    return [(0, M1 + Wp)], [(s, s + M1) for s in s0s]


def _row_map(L):
    """relative row -> shared row over the rounded intervals (must be unique)."""
    m = {}
    for a, n, sm in zip(L["start"], L["len"], L["smem"]):
        for x in range(n):
            assert a + x not in m, f"relative row {a + x} staged twice"
            m[a + x] = sm + x
    return m


def _check_layout(kind, T, W, alpha, base="fib", K=15, dedup=True):
    f = fa.base(base, K)
    L = fa.staging_layout(kind, T, W, alpha, f, dedup=dedup)
    p = fa.rung_params(np.float32(alpha), f, W, dedup=dedup)
    staged = p["active"] & (p["d"] <= T - 1)
    # shared rows: intervals back to back, whole 8-row copies
    assert L["smem"][0] == 0 and np.all(L["len"] % 8 == 0)
    assert np.all(L["smem"][1:] == (L["smem"] + L["len"])[:-1])
    assert np.all(np.diff(L["start"]) > 0)
    m = _row_map(L)
    band, slabs = _ranges(kind, W, [int(s) for s in p["s0"]])
    for a, b in band:
        rows = [m.get(x, -1) for x in range(a, b)]
        assert rows == list(range(rows[0], rows[0] + (b - a))) and rows[0] >= 0
    for k, (a, b) in enumerate(slabs):
        if not staged[k]:
            assert L["slab_row"][k] == -1
            continue
        rows = [m.get(x, -1) for x in range(a, b)]
        assert rows[0] == L["slab_row"][k], (kind, T, alpha, k)
        assert rows == list(range(rows[0], rows[0] + (b - a))), (kind, T, alpha, k, rows[:5])


@pytest.mark.parametrize("kind", ["query", "key"])
def test_slab_that_starts_in_the_rounding_padding(kind):
    _check_layout(kind, 333, 8, 0.87)            # rung 11 slab 4 rows after interval 0's end


@pytest.mark.parametrize("kind", ["query", "key"])
def test_layouts_over_an_alpha_sweep(kind):
    for T in (1, 77, 333, 1024, 2100, 4096):
        for W in (0, 3, 8, 12, 16):
            for alpha in np.linspace(0.5, 1.5, 41):
                _check_layout(kind, T, W, float(np.float32(alpha)))
    for alpha in np.linspace(0.5, 1.5, 21):      # other bases, no dedup
        _check_layout(kind, 1024, 8, float(alpha), base="pow2", K=10)
        _check_layout(kind, 1024, 4, float(alpha), K=12, dedup=False)


def test_learned_alphas_of_the_bench_stack():
    from paper_2606_28560_gb300 import inputs
    theta = inputs.theta_learned(16, seed=3)
    for a in fa.alpha_schedule("learned", 16, theta=theta):
        for kind in ("query", "key"):
            _check_layout(kind, 1024, 8, float(a))


def test_unsupported_shapes():
    with pytest.raises(fa.FibattnError):
        fa.staging_layout("query", 100, 17, 1.0, fa.base("fib", 15))

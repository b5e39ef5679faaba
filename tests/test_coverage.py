"""Coverage of a layer stack (Section 4.2, "Why staggering widens coverage"):
the oracle's set definition against hand-worked sets, and the library's
fibattn_coverage against the oracle across schedules, bases and windows."""
from __future__ import annotations

import numpy as np
import pytest

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import inputs


def test_oracle_hand_worked_sets():
    # f = 1, 2, 3, 5, 8 at alpha = 1.5, W = 2: d = 1.5, 3, 4.5, 7.5, 12.  Dedup
    # drops 1.5; 3 and 12 are integer (one row each), 4.5 and 7.5 read two rows:
    # D = {0,1,2} + {3} + {4,5} + {7,8} + {12}.
    c = O.coverage([1.5], [1, 2, 3, 5, 8], W=2, T=100)
    assert c["per_layer"] == [9] and c["union"] == 9 and c["beyond_window"] == 6
    # without dedup 1.5 adds {1, 2}: already in the window
    assert O.coverage([1.5], [1, 2, 3, 5, 8], W=2, T=100, dedup=False)["union"] == 9
    # reach: at T = 8 no query reaches d = 7.5 or 12 (d > T-1)
    c = O.coverage([1.5], [1, 2, 3, 5, 8], W=2, T=8)
    assert c["union"] == 6                       # {0,1,2,3,4,5}
    # two hops over a pair of layers with D = {0, 1, 3}: sums {0,1,2,3,4,6}
    assert O.coverage([1.0, 1.0], [3], W=1, T=20)["two_hop"] == 6
    # no rungs / one position
    assert O.coverage([1.0], [], W=5, T=64)["union"] == 6
    assert O.coverage([1.0], [1, 2, 3], W=0, T=1)["union"] == 1


def test_fixed_schedule_reads_nineteen_distances():
    """At alpha = 1 (integer rungs) with W = 8 and T = 1024 a layer reads the 9
    window distances and the 10 Fibonacci rungs 13 .. 987 -- the paper's
    "about 19" counted with the window -- and every layer the same ones."""
    f = fa.base("fib", 15)
    c = O.coverage([1.0] * 16, f, W=8, T=1024)
    assert c["per_layer"] == [19] * 16 and c["union"] == 19 and c["beyond_window"] == 10


@pytest.mark.parametrize("kind", ["fixed", "linear", "coprime", "learned"])
@pytest.mark.parametrize("base,K", [("fib", 15), ("pow2", 10)])
@pytest.mark.parametrize("W,T", [(6, 1024), (8, 1024), (12, 1024), (10, 4096)])
def test_library_matches_oracle(kind, base, K, W, T):
    th = inputs.theta_learned(16, seed=3) if kind == "learned" else None
    alphas = fa.alpha_schedule(kind, 16, theta=th)
    f = fa.base(base, K)
    got = fa.coverage(alphas, f, W, T)
    ref = O.coverage(alphas, f, W, T)
    np.testing.assert_array_equal(got["per_layer"], ref["per_layer"])
    for key in ("union", "beyond_window", "two_hop"):
        assert got[key] == ref[key], key


def test_staggering_widens_the_union():
    """The linear ramp reads several times the distinct distances of alpha = 1."""
    f = fa.base("fib", 15)
    fixed = fa.coverage(fa.alpha_schedule("fixed", 16), f, 8, 1024)
    ramp = fa.coverage(fa.alpha_schedule("linear", 16), f, 8, 1024)
    assert ramp["beyond_window"] >= 4 * fixed["beyond_window"]
    assert ramp["two_hop"] > fixed["two_hop"]


def test_coverage_rejects_bad_arguments():
    with pytest.raises(fa.FibattnError):
        fa.coverage([], [1, 2], 4, 64)
    with pytest.raises(fa.FibattnError):
        fa.coverage([1.0], [1, 2], 4, 0)
    with pytest.raises(fa.FibattnError):
        fa.coverage([0.2], [1, 2], 4, 64)          # alpha out of [0.5, 1.5]

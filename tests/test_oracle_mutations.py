"""Plant plausible mistakes in copies of the oracle's C source (CPU only) and
check that the pins catch every one of them."""
from __future__ import annotations

import os
import subprocess

import pytest

import oracle as O
from tests import test_oracle_pins as P

SRC = os.path.join(os.path.dirname(O.__file__), "fibattn_oracle.c")

# (name, original text, planted mistake)
MUTATIONS = [
    ("rope_sign", "y[m + half] = b * c + a * s;", "y[m + half] = b * c - a * s;"),
    ("rope_pairing", "double a = x[m], b = x[m + half];", "double a = x[m], b = x[(m + 1) % half + half];"),
    ("interp_weights_swapped", "sl[n].c0 = 1.0 - w; sl[n].c1 = w;", "sl[n].c0 = w; sl[n].c1 = 1.0 - w;"),
    ("floor_row_index", "int j0 = i - (int)s0;", "int j0 = i - (int)s0 + 1;"),
    ("window_off_by_one", "for (int t = 0; t <= W; ++t) {", "for (int t = 0; t < W; ++t) {"),
    ("mask_boundary", "if (d[k] > (double)i) continue;", "if (d[k] >= (double)i) continue;"),
    ("dedup_boundary", "if (dedup && !(d[k] > (double)W)) continue;", "if (dedup && !(d[k] >= (double)W)) continue;"),
    ("softmax_no_max_shift_in_lse", "if (LSE) LSE[i] = mx + log(l);", "if (LSE) LSE[i] = log(l);"),
    ("dq_missing_scale", "dqt[e] += scale * ds * key[e];", "dqt[e] += ds * key[e];"),
    ("dv_wrong_coeff", "if (sl[s].j1 >= 0) dVp[(size_t)sl[s].j1 * D + e] += sl[s].c1 * gv;",
     "if (sl[s].j1 >= 0) dVp[(size_t)sl[s].j1 * D + e] += sl[s].c0 * gv;"),
    ("dd_value_term_dropped", "acc += pr[s] * dot(go, diff, D);", "acc += 0.0 * dot(go, diff, D);"),
    ("dd_key_sign", "acc += scale * ds * dot(qt, diff, D);", "acc -= scale * ds * dot(qt, diff, D);"),
    ("delta_term", "double ds = pr[s] * (dp[s] - delta);", "double ds = pr[s] * dp[s];"),
    ("inverse_rope_sign", "y[m] = a * c + b * s;", "y[m] = a * c - b * s;"),
    ("dtheta_chain", "*dtheta = da * (alpha - 0.5) * (1.5 - alpha);", "*dtheta = da * (alpha - 0.5);"),
    ("fp32_offsets_skipped", "d_out[k] = (double)(float)((double)a * (double)fk);", "d_out[k] = alpha * f[k];"),
]

PINS = [
    lambda: P.test_integer_alpha_equals_boolean_mask_attention(64, 8, 4, 2, 1),
    lambda: P.test_integer_alpha_equals_boolean_mask_attention(130, 12, 2, 2, 3),
    lambda: P.test_fractional_alpha_equals_interpolation_matrix(0.8125),
    lambda: P.test_backward_equals_autograd_of_matrix_form(0.8125, True),
    lambda: P.test_backward_equals_autograd_of_matrix_form(1.0, True),
    P.test_dtheta_matches_finite_difference,
    P.test_dtheta_nonzero_at_integer_alpha_one_sided,
    lambda: P.test_slot_invariants(0.7333333),
    P.test_rung_exactly_at_position_reads_row_zero,
    P.test_single_position_and_empty_batch,
    P.test_offsets_fp32_rounding,
    P.test_dense_window_is_causal_attention,
]


@pytest.mark.parametrize("name,orig,bad", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_planted_mistake(tmp_path, name, orig, bad):
    src = open(SRC).read()
    assert src.count(orig) == 1, f"mutation anchor for {name} not unique"
    mutated = tmp_path / "mut.c"
    mutated.write_text(src.replace(orig, bad))
    so = tmp_path / "libmut.so"
    subprocess.run(["gcc", "-O2", "-ffp-contract=off", "-fopenmp", "-shared", "-fPIC", "-o", str(so),
                    str(mutated), "-lm"], check=True)
    prev = O._swap_library(str(so))
    caught = []
    try:
        for pin in PINS:
            try:
                pin()
            except (AssertionError, ValueError, FloatingPointError):
                caught.append(pin)
    finally:
        O._swap_library(prev)
    assert caught, f"no pin caught the planted mistake {name!r}"

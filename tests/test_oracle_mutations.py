"""Planted mistakes: each edit below is a plausible slip in the oracle.  Built
into a scratch library, every one must make at least one pin fail -- evidence
that the pins constrain the oracle rather than merely re-run it."""
import numpy as np
import pytest

import oracle
import test_oracle_formats as F
import test_oracle_sweep as SW

MUTATIONS = [
    ("rne-ties-up", "if (d < bd || (d == bd && (k % 2) == 0)) {\n            best = k;",
     "if (d < bd || (d == bd)) {\n            best = k;", [F.test_e2m1_rne_bruteforce]),
    ("loss-drops-weight", "L += wi * e * e;", "L += e * e;", [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("loss-sign", "double e = (double)y[i] - q * v;", "double e = (double)y[i] + q * v;",
     [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("t-uses-v-not-r", "float t = y[i] * r;", "float t = y[i] * vf;", [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("normalise-by-division", "y[i] = usable ? xb[i] * E : xb[i];", "y[i] = usable ? xb[i] / S : xb[i];",
     [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("window-top-6", "chi = clampi(I0 + win_hi, 1, 126);", "chi = clampi(I0 + win_hi - 1, 1, 126);",
     [SW.test_window_edge_blocks]),
    ("window-bottom-shift", "clo = clampi(I0 + win_lo, 1, 126);", "clo = clampi(I0 + win_lo + 1, 1, 126);",
     [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("I0-rounds", "int I0 = oracle_e4m3_floor(sbase);", "int I0 = oracle_e4m3_rn(sbase);",
     [SW.test_bruteforce_matches_oracle_small_blocks]),
    ("ties-to-highest-code", "if (L < Lbest) {\n                        Lsecond = Lbest;",
     "if (L <= Lbest) {\n                        Lsecond = Lbest;", [SW.test_single_spike_block]),
    ("absmax-floor", "int c6 = oracle_e4m3_rn(sbase);", "int c6 = oracle_e4m3_floor(sbase);",
     [SW.test_absmax_and_four_six_scales_use_rn]),
    ("four-six-uses-m-over-3", "float s4 = m / 4.0f;", "float s4 = m / 3.0f;", [SW.test_absmax_and_four_six_scales_use_rn]),
    ("dequant-no-S", "float xh = qv * S;", "float xh = qv;", [SW.test_dequantize_matches_format_tables]),
    ("global-scale-4D", "float sixD = 6.0f * D;", "float sixD = 4.0f * D;", [SW.test_global_scale_planted_max]),
    ("e4m3-bias-6", "int bias = (1 << (e - 1)) - 1;", "int bias = (1 << (e - 1)) - 2 + (e == 2);",
     [F.test_e4m3_facts]),
    ("swizzle-transposed", "(r % 32) * 16 + ((r / 32) % 4) * 4", "(r % 32) * 4 + ((r / 32) % 4) * 16",
     [lambda o: SW.test_swizzle_layout_structure(o, 256, 8)]),
    ("nan-block-swept", "if (isnan(a)) has_nan = 1;", "if (isnan(a)) has_nan = 0;",
     [SW.test_nonfinite_and_out_of_range_blocks]),
    ("no-2^48-bound", "!(m < 0x1p48f)", "!(m < INFINITY)", [SW.test_nonfinite_and_out_of_range_blocks]),
    ("fp8-opt-floor-only", "if (Lc < Lf) { *code = ce;", "if (0) { *code = ce;",
     [SW.test_fp8_quantised_optimum_picks_better_of_floor_and_ceil]),
    ("fp8-opt-ceil-only", "if (Lc < Lf) { *code = ce;", "if (1) { *code = ce;",
     [SW.test_fp8_quantised_optimum_picks_better_of_floor_and_ceil]),
    ("fp8-opt-ties-to-ceil", "if (Lc < Lf) { *code = ce;", "if (Lc <= Lf) { *code = ce;",
     [SW.test_fp8_quantised_optimum_picks_better_of_floor_and_ceil]),
    ("opt-scale-wrong-midpoint", "{0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0}", "{0.25, 0.75, 1.25, 1.75, 2.5, 3.0, 5.0}",
     [SW.test_opt_scale_against_dense_scan]),
]


@pytest.mark.parametrize("name,old,new,pins", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, name, old, new, pins):
    src = oracle.source_text()
    assert src.count(old) >= 1, f"mutation anchor missing: {name}"
    path = oracle.build_variant(src.replace(old, new, 1), str(tmp_path / f"lib_{name}.so"))
    prev = oracle.swap_library(path)
    try:
        caught = False
        for pin in pins:
            try:
                pin(oracle)
            except AssertionError:
                caught = True
        assert caught, f"planted mistake {name} passed every pin"
    finally:
        oracle.swap_library(None)
        oracle._lib = prev

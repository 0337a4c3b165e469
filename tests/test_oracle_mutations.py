"""The pins must catch plausible mistakes in the oracle.  Each case copies the
oracle source to a temporary directory, plants one mistake there (a dropped
term, a wrong sign, a transposed operand, an off-by-one, a wrong tie rule),
builds the copy and checks that at least one pin fails on it.  The committed
oracle is never modified."""
import os

import pytest
import torch

import oracle
import test_oracle_bruteforce as tb
import test_oracle_closed_forms as tc
import test_oracle_decoders as td
import test_oracle_golden as tg
import test_oracle_predicate as tp
import test_oracle_forensics as tf
import test_oracle_stats as ts
from _golden import fixture_files

SRC = os.path.join(os.path.dirname(oracle.__file__), "nmv_oracle.c")

MUTATIONS = {
    "plus_becomes_minus": ("double allowed = atol + scaled;", "double allowed = atol - scaled;"),
    "scale_by_cand": ("double scaled = rtol * fabs(r);", "double scaled = rtol * fabs(c);"),
    "strict_boundary": ("return err <= allowed;", "return err < allowed;"),
    "drop_equality_clause": ("if (c == r) return 1;", ""),
    "nan_passes_as_equal": ("if (c == r) return 1;", "if (c == r || (isnan(c) && isnan(r))) return 1;"),
    "argmax_last_tie": ("if (arg_abs < 0 || a > max_abs)", "if (arg_abs < 0 || a >= max_abs)"),
    "rel_by_cand": ("double rel = a / fabs(r);", "double rel = a / fabs(c);"),
    "rel_includes_zero_ref": ("if (r != 0.0) {", "if (1) {"),
    "drop_compensation": ("if (fabs(sse_sum) >= fabs(term)) sse_comp += (sse_sum - t) + term;",
                          "if (fabs(sse_sum) >= fabs(term)) sse_comp += 0.0;"),
    "transposed_tile_index": ("tile_hist[(row / tile_rows) * grid_cols + col / tile_cols]",
                              "tile_hist[(col / tile_cols) * grid_rows + row / tile_rows]"),
    "row_profile_wrong_index": ("row_prof[row % tile_rows] += 1;",
                                "row_prof[(row / tile_rows) % tile_rows] += 1;"),
    "f16_subnormal_scale": ("v = ldexp((double)frac, -24);", "v = ldexp((double)frac, -25);"),
    "bf16_bias": ("v = ldexp((double)(128u + frac), (int)expo - 134);",
                  "v = ldexp((double)(128u + frac), (int)expo - 133);"),
    "passthrough_without_ref_exclusion": ("if (cb == xb && rb != xb)", "if (cb == xb)"),
    "constant_single_element": ("if (numel >= 2 && cand_constant)", "if (numel >= 1 && cand_constant)"),
    "finite_set_ignores_ref": ("if (isfinite(c) && isfinite(r)) {", "if (isfinite(c)) {"),
    "all_zero_by_bits": ("if (!(c == 0.0)) cand_all_zero = 0;", "if (cb != 0) cand_all_zero = 0;"),
    "threshold_floor": ("int64_t threshold = (numel + 99) / 100;", "int64_t threshold = numel / 100;"),
    "first_k_one_short": ("if (k_out < first_k) {", "if (k_out + 1 < first_k) {"),
    # diagnostic tensor statistics
    "stats_negative_zero_not_zero": ("if (x == 0.0) a->cnt[4]++;", "if (bits == 0) a->cnt[4]++;"),
    "stats_infinities_counted_finite": (
        "if (isinf(x)) { if (x > 0) a->cnt[2]++; else a->cnt[3]++; return; }",
        "if (isinf(x)) { if (x > 0) a->cnt[2]++; else a->cnt[3]++; }"),
    "stats_sample_variance": ("double var = ex2 - mean * mean;",
                              "double var = (ex2 - mean * mean) * n / (n - 1.0);"),
    "stats_tile_transposed": ("int64_t t = tr * gc + tc;", "int64_t t = tc * gr + tr;"),
    "stats_sum_uncompensated": ("f[2] = a->s + a->sc;", "f[2] = a->s;"),
    "stats_int_square_in_32_bits": ("a->iq += (__int128)(v * v);",
                                    "a->iq += (__int128)(int32_t)((int32_t)v * (int32_t)v);"),
    "stats_first_inf_takes_nan": ("if (isinf(v) && first_inf < 0) first_inf = i;",
                                  "if (!isfinite(v) && first_inf < 0) first_inf = i;"),
    "stats_tile_row_overlap": ("r < nrows && r < (tr + 1) * tile_rows; ++r)",
                               "r < nrows && r <= (tr + 1) * tile_rows; ++r)"),
    "stats_min_includes_first_zero": ("if (!a->have || x < a->mn) a->mn = x;",
                                      "if (x < a->mn) a->mn = x;"),
    # deep forensics
    "fx_ulp_from_raw_bits": ("return sign ? -mag : mag;", "return (int64_t)bits;"),
    "fx_ulp_bin_off_by_one": ("while (k < OR_ULP_BINS - 1 && u >= ((int64_t)1 << k)) k++;",
                              "while (k < OR_ULP_BINS - 1 && u > ((int64_t)1 << k)) k++;"),
    "fx_within_strict": ("if (fabs(c - r) <= or_f16_spacing(r)) within++;",
                         "if (fabs(c - r) < or_f16_spacing(r)) within++;"),
    "fx_subnormal_spacing": ("if (fl < -14) fl = -14;", "if (fl < -15) fl = -15;"),
    "fx_first_axis_marginal_lost": ("int64_t coord = rest % shape[a];",
                                    "int64_t coord = rest % shape[a];\n                if (a == 0) coord = 0;"),
    "fx_quarter_rounds_up": ("int64_t q = len / 4;", "int64_t q = (len + 3) / 4;"),
    "fx_near_pass_ignores_nonfinite": ("if (mismatch > 0 && nonfin == 0 && max_ulp <= near_ulps &&",
                                       "if (mismatch > 0 && max_ulp <= near_ulps &&"),
    "fx_growth_axis_stride": ("for (int a = rank - 1; a > axis; --a) stride *= shape[a];",
                              "for (int a = rank - 1; a >= axis; --a) stride *= shape[a];"),
    "fx_argmax_ulp_last": ("if (u > max_ulp) { max_ulp = u; arg_ulp = i; }",
                           "if (u >= max_ulp) { max_ulp = u; arg_ulp = i; }"),
}


def _pins(orc):
    yield lambda: [tg.test_oracle_matches_hand_derived_fixture(orc, p) for p in fixture_files()]
    yield lambda: tp.test_special_value_table(orc)
    yield lambda: tp.test_exact_atol_boundary(orc)
    yield lambda: tp.test_exact_rtol_boundary(orc)
    yield lambda: tb.test_sse_is_compensated(orc)
    yield lambda: [tb.test_fuzz_against_brute_force(orc, s) for s in range(60)]
    yield lambda: [tp.test_matches_torch_isclose_random(orc, dt, s)
                   for dt in (torch.float32, torch.int32) for s in range(2)]
    yield lambda: tc.test_c4_closed_form(orc, 1 << 16)
    yield lambda: tc.test_c1_closed_form(orc)
    yield lambda: td.test_decode_f16_exhaustive(orc)
    yield lambda: td.test_decode_bf16_exhaustive(orc)
    yield lambda: [ts.test_stats_fuzz_against_brute_force(orc, s) for s in range(60)]
    yield lambda: [ts.test_stats_arithmetic_sequence(orc, dt) for dt in (torch.int32, torch.float32)]
    yield lambda: ts.test_stats_constant_and_specials(orc)
    yield lambda: ts.test_stats_int32_sums_are_exact(orc)
    yield lambda: ts.test_stats_float_sums_are_compensated(orc)
    yield lambda: ts.test_stats_empty_and_rank0(orc)
    yield lambda: [tf.test_forensics_fuzz_against_brute_force(orc, s) for s in range(60)]
    yield lambda: tf.test_forensics_ulp_distances_by_hand(orc)
    yield lambda: tf.test_forensics_f16_spacing_boundary(orc)
    yield lambda: tf.test_forensics_growth_and_marginals_closed_form(orc)
    yield lambda: tf.test_forensics_near_pass(orc)


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(tmp_path, name):
    before, after = MUTATIONS[name]
    text = open(SRC).read()
    assert text.count(before) == 1, "mutation anchor must be unique: %r" % before
    src = tmp_path / "mutant.c"
    src.write_text(text.replace(before, after))
    lib = oracle.build(force=True, src=str(src), out=str(tmp_path / "libmutant.so"))
    orc = oracle.Oracle(lib)
    for pin in _pins(orc):
        try:
            pin()
        except (AssertionError, ValueError, IndexError):
            return
    pytest.fail("no pin caught the planted mistake %r" % name)

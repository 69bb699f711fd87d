"""Plant plausible mistakes in copies of oracle.c and check the pins catch
each one (the mistakes live only in temporary copies, on the CPU).

Each mutant is a one-line edit of the kind a hand-written oracle could
contain: a dropped term, a wrong sign or index, a transposed operand, a
lost precision, a wrong tie-break, a wrong fill value.
"""
import os

import pytest

import oracle as default_oracle
from test_oracle_pins import PINS
from test_oracle_sampling import SAMPLING_PINS
from test_oracle_fp8 import FP8_PINS
from test_oracle_recall import RECALL_PINS

SRC = os.path.join(os.path.dirname(default_oracle.__file__), "oracle.c")

MUTANTS = {
    "dropped_first_term": ("for (int32_t j = 0; j < d; ++j)", "for (int32_t j = 1; j < d; ++j)"),
    "dropped_last_term": ("for (int32_t j = 0; j < d; ++j)", "for (int32_t j = 0; j + 1 < d; ++j)"),
    "wrong_sort_sign": ("if (a->z > b->z) return -1;\n    if (a->z < b->z) return 1;",
                        "if (a->z < b->z) return -1;\n    if (a->z > b->z) return 1;"),
    "reversed_tie_break": ("if (a->i < b->i) return -1;\n    if (a->i > b->i) return 1;",
                           "if (a->i > b->i) return -1;\n    if (a->i < b->i) return 1;"),
    "transposed_weight": ("acc += oracle_bf16_to_double(wi[j]) * (double)hb[j];",
                          "acc += oracle_bf16_to_double(W[(int64_t)j * V + i]) * (double)hb[j];"),
    "reversed_query_index": ("acc += oracle_bf16_to_double(wi[j]) * (double)hb[j];",
                             "acc += oracle_bf16_to_double(wi[j]) * (double)hb[d - 1 - j];"),
    "bf16_wrong_shift": ("uint32_t u = ((uint32_t)bits) << 16;", "uint32_t u = ((uint32_t)bits) << 15;"),
    "fp32_accumulator": ("double acc = 0.0;", "float acc = 0.0f;"),
    "unsorted_logit_copy": ("logits[(int64_t)b * k + j] = rows[j].z;", "logits[(int64_t)b * k + j] = z[j];"),
    "zero_fill_not_neg_inf": ("row[v] = -INFINITY;", "row[v] = 0.0f;"),
    "no_range_check": ("if (t < 0 || (int64_t)t >= V) {", "if (t < 0) {"),
    # top-k sampling and its generator
    "philox_wrong_multiplier": ("(uint64_t)0xD2511F53u * c0", "(uint64_t)0xD2511F55u * c0"),
    "philox_key_not_bumped": ("k1 += 0xBB67AE85u;", "k1 += 0u;"),
    "philox_words_swapped": ("const uint32_t n1 = (uint32_t)p1;", "const uint32_t n1 = (uint32_t)p0;"),
    "uniform_wrong_bits": ("(double)(out[0] >> 8) * (1.0 / 16777216.0)", "(double)(out[1] >> 8) * (1.0 / 16777216.0)"),
    "temperature_dropped": ("p[j] = exp(z[j] / T - s0);", "p[j] = exp(z[j] - s0);"),
    "top_p_strict": ("if (run >= top_p) {", "if (run > top_p) {"),
    "min_p_absolute": ("if (p[j] >= min_p * p[0]) ++n_m;", "if (p[j] >= min_p) ++n_m;"),
    "draw_at_or_above": ("if (cum > target) {", "if (cum >= target) {"),
    "prob_not_renormalised": ("*prob_out = p[js] / M;", "*prob_out = p[js];"),
    # the quantised head
    "e4m3_truncated": ("double m = rint((ldexp(a, -e) - 1.0) * 8.0);", "double m = floor((ldexp(a, -e) - 1.0) * 8.0);"),
    "e4m3_bias_off": ("return (uint8_t)((sgn << 7) | ((e + 7) << 3) | (int)m);", "return (uint8_t)((sgn << 7) | ((e + 8) << 3) | (int)m);"),
    "e4m3_subnormal_step": ("const double m = rint(ldexp(a, 9));", "const double m = rint(ldexp(a, 8));"),
    "e4m3_decode_bias": ("v = ldexp(1.0 + M / 8.0, E - 7);", "v = ldexp(1.0 + M / 8.0, E - 8);"),
    "scale_wrong_range": ("const float s = amax > 0.0f ? amax / 448.0f : 1.0f;", "const float s = amax > 0.0f ? amax / 240.0f : 1.0f;"),
    "logits_scale_dropped": ("zb[i] = (double)scale[i] * acc;", "zb[i] = acc;"),
    # Recall@k bookkeeping
    "recall_repeats_counted": ("++h;\n                    break;", "++h;"),
    "recall_last_candidate_missed": ("for (int32_t i = 0; i < m; ++i) {", "for (int32_t i = 0; i + 1 < m; ++i) {"),
    "recall_wrong_row_stride": ("*aq = approx + q * m;", "*aq = approx + q * k;"),
    "recall_empty_slots_match": ("if (eq[j] < 0) continue;", ""),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTANTS[name]
    text = open(SRC).read()
    assert text.count(old) >= 1, f"mutation site for {name} not found"
    src = tmp_path / f"oracle_{name}.c"
    src.write_text(text.replace(old, new, 1))
    lib = default_oracle.OracleLib(default_oracle.build(True, str(src), str(tmp_path / f"{name}.so")))
    caught = []
    for pin_name, pin in PINS + SAMPLING_PINS + FP8_PINS + RECALL_PINS:
        try:
            pin(lib)
        except (AssertionError, ValueError):
            caught.append(pin_name)
    assert caught, f"no pin caught mutant {name}"

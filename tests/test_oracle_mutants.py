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
    for pin_name, pin in PINS:
        try:
            pin(lib)
        except (AssertionError, ValueError):
            caught.append(pin_name)
    assert caught, f"no pin caught mutant {name}"

"""The oracle pins must reject plausible mistakes.

Each case plants one mistake in a temporary copy of oracle/dkv_oracle.c (an
off-by-one bin, a reversed distance, a wrong window edge, intersection instead of
union, strided GQA grouping, a dropped scale, swapped operands, offsets without
the reserve, appending at the wrong slot, Top-K ties or order reversed, a
truncating budget), builds it with the host C compiler,
and runs the pin suite against it: at least one pin has to fail. The real oracle
is restored afterwards. CPU only.
"""
import os
import subprocess
import sys
import tempfile

import pytest

import oracle as O
import test_oracle_pins as pins
from golden_io import map_cases

SRC = os.path.join(os.path.dirname(O.__file__), "dkv_oracle.c")

MUTANTS = {
    "bin_off_by_one": ("return (Tc - (long)s->recent - 1 - p) / (long)s->bin_width;",
                       "return (Tc - (long)s->recent - p) / (long)s->bin_width;"),
    "bin_from_start": ("return (Tc - (long)s->recent - 1 - p) / (long)s->bin_width;",
                       "return (p - (long)s->sink) / (long)s->bin_width;"),
    "recent_edge": ("if (p >= Tc - (long)s->recent) return 1;",
                    "if (p > Tc - (long)s->recent) return 1;"),
    "sink_edge": ("if (p < (long)s->sink) return 1;",
                  "if (p <= (long)s->sink) return 1;"),
    "intersection": ("if (oracle_keep_logical(M, s, layer, g * G + j, p, Tc)) return 1;\n    return 0;",
                     "if (!oracle_keep_logical(M, s, layer, g * G + j, p, Tc)) return 0;\n    return 1;"),
    "strided_groups": ("oracle_keep_logical(M, s, layer, g * G + j, p, Tc)",
                       "oracle_keep_logical(M, s, layer, g + j * s->Hkv, p, Tc)"),
    "no_scale": ("sc[r] = scale * dot;", "sc[r] = dot;"),
    "values_as_keys": ("dot += bf16_to_double(qj[k]) * bf16_to_double(Krows[(size_t)r * hd + k]);",
                       "dot += bf16_to_double(qj[k]) * bf16_to_double(Vrows[(size_t)r * hd + k]);"),
    "offsets_without_reserve": ("row += (int64_t)n + reserve;", "row += (int64_t)n;"),
    "append_overwrites_last": ("size_t dst = (size_t)(off[h] + len[h] + na) * hd;",
                               "size_t dst = (size_t)(off[h] + len[h] + na - 1) * hd;"),
    "descending_pack": ("for (long p = 0; p < Tc[b]; ++p)",
                        "for (long p = Tc[b] - 1; p >= 0; --p)"),
    "topk_ties_to_higher_index": ("    return i < j;\n}", "    return i > j;\n}"),
    "topk_nan_first": ("if (na != nb) return nb; /* the number comes first */",
                       "if (na != nb) return na;"),
    "topk_smallest": ("if (!na && a != b) return a > b;", "if (!na && a != b) return a < b;"),
    "budget_truncates": ("(double)D + 0.5);", "(double)D);"),
}


def _pin_calls():
    calls = []
    for Tc, D in [(130816, 1013), (32512, 245)]:
        calls.append(lambda Tc=Tc, D=D: pins.test_bin_count_matches_appendix_a(Tc, D))
    for case in map_cases():
        calls.append(lambda case=case: pins.test_map_hand_worked_cases(case))
    for seed in range(6):
        calls.append(lambda seed=seed: pins.test_length_closed_form(seed))
    for seed in range(4):
        calls.append(lambda seed=seed: pins.test_topk_matches_pairwise_rank_definition(seed))
    for G, hd in [(1, 4), (2, 8), (4, 128), (7, 128)]:
        calls.append(lambda G=G, hd=hd: pins.test_compacted_attention_equals_masked_dense(G, hd))
    for name in ("test_memory_arithmetic_sec43_and_app_c", "test_streaming_llm_special_case",
                 "test_all_keep_is_dense", "test_head_level_special_case",
                 "test_gqa_union_of_query_head_sets", "test_indices_ascending_unique_in_range",
                 "test_compact_is_ordered_gather", "test_all_keep_attention_is_dense_attention",
                 "test_single_row_returns_that_value_row", "test_identical_keys_give_mean_of_values",
                 "test_softmax_weights_sum_to_one_and_two_row_closed_form",
                 "test_default_scale_is_inverse_sqrt_head_dim",
                 "test_append_then_decode_equals_attention_with_new_token", "test_budget_rounding_app_a3",
                 "test_topk_equals_stable_library_sort"):
        calls.append(getattr(pins, name))
    return calls


def _run_pins_against(so_path):
    """Child-process body: count failing pins against the library at so_path."""
    O.use_library(so_path)
    failures = 0
    for call in _pin_calls():
        try:
            call()
        except (AssertionError, O.OracleError):
            failures += 1
    return failures


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_planted_mistake(name):
    before, after = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(before) == 1, f"mutation anchor for {name} not found exactly once"
    with tempfile.TemporaryDirectory() as tmp:
        c = os.path.join(tmp, "mutant.c")
        so = os.path.join(tmp, "libmutant.so")
        open(c, "w").write(src.replace(before, after))
        subprocess.check_call([os.environ.get("CC", "gcc"), "-O1", "-std=c11", "-fPIC", "-shared",
                               "-o", so, c, "-lm"])
        here = os.path.dirname(os.path.abspath(__file__))
        code = ("import sys; sys.path[:0] = [%r, %r]; import test_oracle_mutants as t; "
                "print('FAILED_PINS', t._run_pins_against(%r))" % (here, os.path.dirname(here), so))
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)
    if r.returncode == 0:
        n = int(r.stdout.strip().split()[-1])
        assert n > 0, f"no pin caught the planted mistake {name!r}"
    else:
        # The mutant broke the oracle badly enough to crash the pin run: caught.
        assert r.returncode != 0

"""The oracle's pins are strong enough to catch plausible mistakes.

Each case plants one mistake in a temporary copy of oracle/rr_oracle.c (the
committed oracle is never touched), builds it, points the oracle module at the
mutant and runs the pin checks of test_oracle_pins.py: at least one must fail.
"""
import ctypes
import os
import shutil
import subprocess

import pytest

import oracle
import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "rr_oracle.c")

MUTANTS = {
    "dropped_scale": ("s[j] = scale * dot;", "s[j] = dot;"),
    "wrong_sign_in_exp": ("s[j] = exp(s[j] - m);", "s[j] = exp(m - s[j]);"),
    "gqa_interleaved": ("int32_t h = g * G + hh;", "int32_t h = hh * J->Hkv + g;"),
    "page_index_swapped": ("J->page_table[(int64_t)b * J->max_pages + j / J->ps]",
                           "J->page_table[(int64_t)b * J->max_pages + j % J->ps]"),
    "slot_index_wrong": ("int64_t base = ((page * J->ps + j % J->ps) * J->Hkv + g)",
                         "int64_t base = ((page * J->ps + (J->ps - 1 - j % J->ps)) * J->Hkv + g)"),
    "dims_reversed": ("dot += qv[d] * K[j * D + d];", "dot += qv[d] * K[j * D + (D - 1 - d)];"),
    "values_are_keys": ("o[d] += s[j] * V[j * D + d];", "o[d] += s[j] * K[j * D + d];"),
    "unnormalised": ("for (int32_t d = 0; d < D; ++d) o[d] /= l;", "for (int32_t d = 0; d < D; ++d) o[d] /= l + 1.0;"),
    "causal_strict": ("s[j] = exp(s[j] - m);\n        l += s[j];", "s[j] = j < p ? exp(s[j] - m) : 0.0;\n        l += s[j];"),
    "append_ignores_row_offset": ("int64_t src = (cu + j) * row;", "int64_t src = j * row;"),
    "append_slot_from_row": ("int64_t slot = pos % ps;", "int64_t slot = j % ps;"),
}

CHECKS = [
    lambda: [pins.test_oracle_matches_dense_brute_force(c) for c in pins.CASES],
    pins.test_single_visible_key_returns_value_exactly,
    pins.test_zero_scale_gives_running_mean_of_visible_values,
    pins.test_unit_values_give_unit_output,
    pins.test_two_keys_by_hand,
    pins.test_query_aligned_with_one_key_selects_its_value,
    pins.test_gqa_reads_kv_head_h_div_g,
    pins.test_prefix_extend_equals_full_causal_attention,
    pins.test_page_permutation_is_bit_invariant,
    pins.test_append_gather_back_and_untouched_slots,
    pins.test_append_hand_built_case,
]


def _build_mutant(tmp_path, name):
    old, new = MUTANTS[name]
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation site for {name} not unique"
    src = tmp_path / f"{name}.c"
    src.write_text(text.replace(old, new))
    so = tmp_path / f"{name}.so"
    subprocess.run(["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-std=c11", str(src), "-o", str(so), "-lm"],
                   check=True)
    return str(so)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(tmp_path, monkeypatch, name):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    so = _build_mutant(tmp_path, name)
    real = oracle.lib()
    mutant = ctypes.CDLL(so)
    for fn in ("oracle_kv_append", "oracle_extend_attention", "oracle_attention_rows"):
        getattr(mutant, fn).restype = getattr(real, fn).restype
        getattr(mutant, fn).argtypes = getattr(real, fn).argtypes
    monkeypatch.setattr(oracle, "_lib", mutant)
    caught = []
    for check in CHECKS:
        try:
            check()
        except (AssertionError, oracle.OracleError):
            caught.append(check)
    assert caught, f"no pin caught the planted mistake '{name}'"

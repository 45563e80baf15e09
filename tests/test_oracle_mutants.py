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
import test_oracle_rope_pins as rpins

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
    "rope_sign_of_one_term": ("yr[i] = xr[i] * c - xr[i + half] * s;", "yr[i] = xr[i] * c + xr[i + half] * s;"),
    "rope_turns_backwards": ("yr[i] = xr[i] * c - xr[i + half] * s;\n                yr[i + half] = xr[i + half] * c + xr[i] * s;",
                             "yr[i] = xr[i] * c + xr[i + half] * s;\n                yr[i + half] = xr[i + half] * c - xr[i] * s;"),
    "rope_pairs_mirrored": ("yr[i] = xr[i] * c - xr[i + half] * s;\n                yr[i + half] = xr[i + half] * c + xr[i] * s;",
                            "yr[i] = xr[i] * c - xr[D - 1 - i] * s;\n                yr[D - 1 - i] = xr[D - 1 - i] * c + xr[i] * s;"),
    "rope_frequency_exponent": ("pow(base, -2.0 * i / D)", "pow(base, -1.0 * i / D)"),
    "rope_position_off_by_one": ("(double)pos[r] * pow", "(double)(pos[r] + 1) * pow"),
    "round_truncates": ("ldexp(rint(ldexp(v, -q)), q)", "ldexp(trunc(ldexp(v, -q)), q)"),
    "round_twice_via_float": ("ldexp(rint(ldexp(v, -q)), q)", "ldexp(rint(ldexp((double)(float)v, -q)), q)"),
    "round_no_subnormals": ("if (q < -133) q = -133;", "if (q < -126) q = -126;"),
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
    rpins.test_round_bf16_hand_cases,
    rpins.test_round_bf16_matches_integer_trick_on_float32,
    rpins.test_round_bf16_is_nearest_brute_force,
    rpins.test_rope_position_zero_is_identity,
    rpins.test_rope_keeps_every_pair_length,
    rpins.test_rope_d2_is_the_plane_rotation_by_p_radians,
    lambda: [rpins.test_rope_unit_vector_stays_in_its_pair_and_turns_towards_the_upper_half(D) for D in (8, 64, 128)],
    rpins.test_rope_frequencies_by_hand,
    rpins.test_rope_composes,
    rpins.test_rope_scores_depend_on_relative_position_only,
    rpins.test_rope_append_keeps_position_zero_and_values_bit_exact,
    lambda: [rpins.test_rope_attention_matches_dense_brute_force(sd) for sd in (21, 22)],
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
    for fn in ("oracle_kv_append", "oracle_extend_attention", "oracle_attention_rows", "oracle_extend_attention_q64",
               "oracle_attention_rows_q64", "oracle_rope", "oracle_round_bf16"):
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

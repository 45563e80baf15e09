"""The per-element parity bar of the GPU tests (tests/parity.py), pinned on the CPU.

The bar is 1e-2, plus half a bf16 unit in the last place of the reference where |ref| >= 2: bf16 keeps 8
significant bits, so half a unit is 2^-7 on [2, 4), 2^-6 on [4, 8) and 2^-5 on [8, 16).
"""
import numpy as np
import pytest

from parity import MAX_ABS, max_abs_bar


def test_bar_below_two_is_the_plain_bar():
    for x in (0.0, 1e-30, -0.5, 1.0, 1.999, -1.9999999):
        assert max_abs_bar(np.array([x]))[0] == MAX_ABS


def test_bar_adds_half_a_unit_in_the_last_place():
    cases = [(2.0, 2.0 ** -7), (-3.99, 2.0 ** -7), (4.0, 2.0 ** -6), (-6.0, 2.0 ** -6), (7.999, 2.0 ** -6),
             (8.0, 2.0 ** -5), (15.0, 2.0 ** -5)]
    for x, half in cases:
        assert max_abs_bar(np.array([x]))[0] == MAX_ABS + half, x
        assert max_abs_bar(np.array([x]))[0] - MAX_ABS == pytest.approx(half, rel=1e-12)


def test_half_unit_matches_the_spacing_of_bf16():
    # the spacing of bf16 numbers on [2^e, 2^(e+1)) is 2^(e-7): step from 1 + 2^-7 (the first bf16 above 1)
    for e in range(1, 6):
        lo = 2.0 ** e
        nxt = lo * (1 + 2.0 ** -7)
        assert max_abs_bar(np.array([lo]))[0] - MAX_ABS == pytest.approx((nxt - lo) / 2, rel=1e-12)

"""Pins of the oracle's rotary position embedding and bf16 rounding (CPU only).

The paper never writes positional encodings; the reading (rotate-half pairing, angle p * base^(-2i/D),
RoFormer's rotation direction) is stated in section (C) of oracle/rr_oracle.c.  Each pin checks it
against something other than the oracle's own formula:

* bf16 rounding: bit patterns fixed by the format (1.0 = 0x3F80, ties to even, one rounding from the
  double, subnormals), the integer round-to-nearest-even trick on binary32 bits for float32 inputs,
  and brute-force nearness against both neighbouring bf16 values;
* rotation: position 0 is the identity; each (i, i + D/2) pair keeps its length; D = 2 is the plane
  rotation by p radians (complex multiplication by e^(ip)); a unit vector stays in its own pair and
  turns towards + the upper half; the frequency of pair i worked out by hand for D = 8, base 10^4;
  rotations compose (p then q equals p + q); scores depend on the relative position only;
* rotated extend attention and rotated decode against a dense brute force that rotates through
  complex numbers and masks with an explicit matrix; a P = 0 agent's first key is stored unrotated,
  bit for bit.
"""
import math

import numpy as np
import pytest

import oracle
import synth


# ------------------------------------------------------------------ bf16 rounding

def test_round_bf16_hand_cases():
    one = 0x3F80  # sign 0, biased exponent 127, fraction 0
    cases = [
        (1.0, one),
        (1.0 + 2.0 ** -8, one),                            # halfway between 1 and 1 + 2^-7: tie -> even (1)
        (1.0 + 3 * 2.0 ** -8, one + 2),                    # halfway between 1 + 2^-7 and 1 + 2^-6: -> even
        (1.0 + 2.0 ** -8 + 2.0 ** -40, one + 1),           # just above the tie
        (1.0 + 2.0 ** -8 + 2.0 ** -30, one + 1),           # one rounding: via float32 it would be a tie -> 1
        (-(1.0 + 2.0 ** -8 + 2.0 ** -40), 0x8000 | (one + 1)),
        (2.0 ** -130, 0x0008),                             # subnormal: 8 x 2^-133
        (2.0 ** -134, 0x0000),                             # half the smallest subnormal: tie -> even (0)
        (3 * 2.0 ** -134, 0x0002),                         # 1.5 x 2^-133: tie -> even (2 x 2^-133)
        (0.0, 0x0000),
        (255.5, 0x437F + 1),                               # 255.5 halfway between 255 and 256 -> even (256)
    ]
    got = oracle.round_bf16(np.array([c[0] for c in cases]))
    assert [int(g) for g in got] == [c[1] for c in cases]


def test_round_bf16_matches_integer_trick_on_float32():
    rng = np.random.default_rng(5)
    f = (rng.standard_normal(200000) * np.exp2(rng.integers(-30, 30, 200000))).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    trick = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    assert np.array_equal(oracle.round_bf16(f.astype(np.float64)), trick)


def test_round_bf16_is_nearest_brute_force():
    rng = np.random.default_rng(6)
    x = rng.standard_normal(50000) * 10.0 ** rng.integers(-3, 4, 50000)
    r = oracle.round_bf16(x)
    val = oracle.widen_bf16(r)
    up = oracle.widen_bf16(r + np.where(x >= 0, 1, -1).astype(np.uint16))   # next bf16 away from zero
    dn = oracle.widen_bf16(r - np.where(x >= 0, 1, -1).astype(np.uint16))   # next bf16 towards zero
    assert (np.abs(x - val) <= np.abs(x - up)).all()
    assert (np.abs(x - val) <= np.abs(x - dn)).all()


# ------------------------------------------------------------------ rotation

def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_rope_position_zero_is_identity():
    x = _rand((5, 3, 128), 1)
    assert np.array_equal(oracle.rope(x, np.zeros(5, np.int64), 500000.0), x)


def test_rope_keeps_every_pair_length():
    x = _rand((40, 2, 64), 2)
    pos = np.random.default_rng(3).integers(0, 300000, 40)
    y = oracle.rope(x, pos, 10000.0)
    h = 32
    np.testing.assert_allclose(y[..., :h] ** 2 + y[..., h:] ** 2, x[..., :h] ** 2 + x[..., h:] ** 2, rtol=1e-12)


def test_rope_d2_is_the_plane_rotation_by_p_radians():
    x = _rand((30, 1, 2), 4)
    pos = np.arange(30) * 7 + 3
    z = (x[:, 0, 0] + 1j * x[:, 0, 1]) * np.exp(1j * pos)
    y = oracle.rope(x, pos, 10000.0)
    np.testing.assert_allclose(y[:, 0, 0], z.real, atol=1e-12)
    np.testing.assert_allclose(y[:, 0, 1], z.imag, atol=1e-12)


@pytest.mark.parametrize("D", [8, 64, 128])
def test_rope_unit_vector_stays_in_its_pair_and_turns_towards_the_upper_half(D):
    h = D // 2
    p = 37
    for j in (0, 1, h - 1):
        x = np.zeros((1, 1, D))
        x[0, 0, j] = 1.0
        y = oracle.rope(x, [p], 10000.0)[0, 0]
        a = p * 10000.0 ** (-2.0 * j / D)
        expect = np.zeros(D)
        expect[j], expect[j + h] = math.cos(a), math.sin(a)
        np.testing.assert_allclose(y, expect, atol=1e-12)
        x = np.zeros((1, 1, D))
        x[0, 0, j + h] = 1.0
        y = oracle.rope(x, [p], 10000.0)[0, 0]
        expect = np.zeros(D)
        expect[j + h], expect[j] = math.cos(a), -math.sin(a)
        np.testing.assert_allclose(y, expect, atol=1e-12)


def test_rope_frequencies_by_hand():
    # D = 8, base 10^4: pair i turns by 10^(-i) radians per position, so at p = 10 the four pairs sit
    # at 10, 1, 0.1 and 0.01 radians
    D, p = 8, 10
    angles = [10.0, 1.0, 0.1, 0.01]
    for i, a in enumerate(angles):
        x = np.zeros((1, 1, D))
        x[0, 0, i] = 1.0
        y = oracle.rope(x, [p], 10000.0)[0, 0]
        assert y[i] == pytest.approx(math.cos(a), abs=1e-13)
        assert y[i + 4] == pytest.approx(math.sin(a), abs=1e-13)


def test_rope_composes():
    x = _rand((12, 2, 64), 7)
    m = np.random.default_rng(8).integers(0, 5000, 12)
    n = np.random.default_rng(9).integers(0, 5000, 12)
    twice = oracle.rope(oracle.rope(x, m, 10000.0), n, 10000.0)
    np.testing.assert_allclose(twice, oracle.rope(x, m + n, 10000.0), atol=1e-9)


def test_rope_scores_depend_on_relative_position_only():
    q = _rand((1, 1, 128), 10)
    k = _rand((1, 1, 128), 11)
    for m, n, c in [(5, 3, 1000), (100, 7, 12345), (0, 0, 65536), (40000, 39000, 3)]:
        s0 = float(np.sum(oracle.rope(q, [m], 500000.0) * oracle.rope(k, [n], 500000.0)))
        s1 = float(np.sum(oracle.rope(q, [m + c], 500000.0) * oracle.rope(k, [n + c], 500000.0)))
        assert s1 == pytest.approx(s0, rel=1e-9, abs=1e-9)


# ------------------------------------------------------------------ rotated append and attention

BASE = 10000.0


def _tiny(seed=21, P=(0, 40, 16), S=(19, 23, 33)):
    P = np.asarray(P, dtype=np.int64)
    S = np.asarray(S, dtype=np.int64)
    return synth.custom("rope_tiny", len(P), 8, 2, 64, P, S, seed=seed)


def test_rope_append_keeps_position_zero_and_values_bit_exact():
    wl = _tiny()
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append_rope(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    kp0, vp0 = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table,
                                wl.prefix_lens, wl.suffix_lens)
    assert np.array_equal(vp, vp0)                      # V is not rotated
    page, slot = wl.page_table[0, 0], 0                 # agent 0 has P = 0: its first key is at position 0
    assert np.array_equal(kp[page, slot], kp0[page, slot])
    assert not np.array_equal(kp, kp0)


def _brute_force_rope(wl, base):
    """Dense rotated attention: rotation through complex numbers, explicit mask, logical keys."""
    t = synth.cpu_tensors(wl)
    q = oracle.widen_bf16(t["q"])
    D, h = wl.D, wl.D // 2
    freq = base ** (-np.arange(h) * 2.0 / D)

    def rot(x, pos):  # x [n, D] or [n, heads, D]
        e = np.exp(1j * np.outer(pos, freq))
        if x.ndim == 3:
            e = e[:, None, :]
        z = (x[..., :h] + 1j * x[..., h:]) * e
        return np.concatenate([z.real, z.imag], axis=-1)

    out = np.zeros(q.shape)
    G = wl.Hq // wl.Hkv
    for b in range(wl.B):
        P, S = int(wl.prefix_lens[b]), int(wl.suffix_lens[b])
        if S == 0:
            continue
        c, L = int(wl.cu[b]), P + S
        pos = P + np.arange(S)
        qr = rot(q[c:c + S], pos)
        mask = np.arange(L)[None, :] <= pos[:, None]
        for g in range(wl.Hkv):
            k, v = synth.agent_kv(wl, b, L, g)
            K, V = oracle.widen_bf16(k), oracle.widen_bf16(v)
            # cached keys as given; the suffix's keys rotated and rounded once to the pool's bf16
            K[P:] = oracle.widen_bf16(oracle.round_bf16(rot(K[P:], pos)))
            for hq in range(g * G, (g + 1) * G):
                s = qr[:, hq, :] @ K.T / math.sqrt(D)
                s = np.where(mask, s, -np.inf)
                w = np.exp(s - s.max(axis=1, keepdims=True))
                out[c:c + S, hq, :] = (w / w.sum(axis=1, keepdims=True)) @ V
    return out


@pytest.mark.parametrize("seed", [21, 22])
def test_rope_attention_matches_dense_brute_force(seed):
    wl = _tiny(seed)
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append_rope(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    got = oracle.extend_attention_rope(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens, BASE)
    np.testing.assert_allclose(got, _brute_force_rope(wl, BASE), atol=1e-11, rtol=0)


def test_rope_attention_single_key_is_value():
    wl = _tiny(P=(0,), S=(1,))
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append_rope(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    got = oracle.extend_attention_rope(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens, BASE)
    v = oracle.widen_bf16(t["v_new"])[0]
    assert np.array_equal(got[0], np.repeat(v, 4, axis=0))


def test_rope_decode_matches_dense_brute_force():
    """Rotated decode (one new token per agent, its query rotated at L - 1) against the same dense brute
    force: the last row of rotated causal attention over the agent's L keys."""
    L = np.array([1, 40, 130])
    wl = synth.custom("rope_dec", 3, 8, 2, 64, L - 1, np.ones(3, dtype=np.int64), seed=23)
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append_rope(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    got = oracle.decode_attention_rope(t["q"], kp, vp, wl.page_table, L.astype(np.int32), BASE)
    np.testing.assert_allclose(got, _brute_force_rope(wl, BASE), atol=1e-11, rtol=0)
    # the one-key agent (position 0: no rotation) returns its value exactly
    v = oracle.widen_bf16(t["v_new"])[0]
    assert np.array_equal(got[0], np.repeat(v, 4, axis=0))


def test_round_bf16_special_values():
    """Values the bf16 format fixes at the ends of its range: the largest finite value 0x7F7F =
    (2 - 2^-7) 2^127; the tie halfway to 2^128 rounds to even, i.e. up to infinity (0x7F80), just below
    it stays finite; signed zero, infinities and NaN (quiet, 0x7FC0) keep their kind."""
    big = (2.0 - 2.0 ** -7) * 2.0 ** 127
    cases = [
        (big, 0x7F7F),
        ((2.0 - 2.0 ** -8) * 2.0 ** 127, 0x7F80),                 # tie above the largest finite value
        ((2.0 - 2.0 ** -8 - 2.0 ** -20) * 2.0 ** 127, 0x7F7F),    # just below the tie
        (-big, 0xFF7F),
        (-0.0, 0x8000),
        (float("inf"), 0x7F80),
        (float("-inf"), 0xFF80),
        (2.0 ** -126, 0x0080),                                     # smallest normal
        (2.0 ** -133, 0x0001),                                     # smallest subnormal
    ]
    got = oracle.round_bf16(np.array([c[0] for c in cases]))
    assert [int(g) for g in got] == [c[1] for c in cases]
    nan = int(oracle.round_bf16(np.array([float("nan")]))[0])
    assert nan & 0x7F80 == 0x7F80 and nan & 0x007F != 0            # a NaN pattern


def test_rope_rejects_odd_head_dim():
    with pytest.raises(oracle.OracleError):
        oracle.rope(np.zeros((2, 1, 7)), [0, 1], 10000.0)

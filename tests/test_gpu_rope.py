"""Rotary position embedding on the GPU (rr_rope_table, rr_kv_append_rope, rr_extend_attention_rope,
rr_extend_step_rope, rr_decode_attention_rope) against the fp64 oracle, on the same seeded inputs.

* the (cos, sin) table against the oracle's rotation of unit vectors (float rounding of the double
  values);
* the rotated append: V and every untouched pool slot bit-exact; each rotated K element within one bf16
  unit in the last place of the oracle's exactly rounded rotation plus the fp32 evaluation error of the
  rotation (the kernel rotates in fp32 from a float table), and almost all of them bit-exact;
* the rotated extend attention within the parity bar of the oracle (q rotated in double precision and
  not rounded; the oracle's own rotated pool): every GQA group, both head dims, prefixes in the middle of
  a page, split-K batches, positions past 10^5 (angles the table must hold to float accuracy);
* the one-call step bit-identical to its two calls; a position past the table reported, and the library
  usable afterwards;
* decode with rotary embedding (q rotated at L_b - 1 by the decode kernel) within the parity bar of the
  oracle: every GQA group, both head dims, split-K, positions past 10^5.
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, to_f64

pytestmark = pytest.mark.gpu

BASE = 500000.0


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def u16(t):
    import torch
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def test_rope_table_matches_oracle_rotation(rr):
    D, max_pos = 128, 300000
    table = rr.rope_table(max_pos, D, BASE).cpu().numpy()
    assert rr.device_error() == 0
    rng = np.random.default_rng(3)
    pos = np.concatenate([[0, 1, 2, 16383, max_pos - 1], rng.integers(0, max_pos, 60)])
    for i in (0, 1, 7, 31, 63):
        e = np.zeros((len(pos), 1, D))
        e[:, 0, i] = 1.0
        y = oracle.rope(e, pos, BASE)[:, 0]       # (cos a, sin a) lands in dims i and i + D/2
        np.testing.assert_allclose(table[pos, i, 0], y[:, i], rtol=0, atol=1.2e-7)
        np.testing.assert_allclose(table[pos, i, 1], y[:, i + D // 2], rtol=0, atol=1.2e-7)


def _within_bound(got_bits, ref_bits):
    """One bf16 unit in the last place, plus the fp32 evaluation error of the rotation.

    The kernel takes cos a and sin a from a float table (each within 2^-24 relative) and rotates in fp32,
    so before its bf16 rounding a result is within a few 2^-24 of the pair's length r = |(x_i, x_i+D/2)|
    (which the rotation keeps) -- many units of a result that nearly cancels.  Bound: 2^-7 of the larger
    value + 2^-21 r."""
    a = oracle.widen_bf16(got_bits)
    b = oracle.widen_bf16(ref_bits)
    h = b.shape[-1] // 2
    r = np.sqrt(b[..., :h] ** 2 + b[..., h:] ** 2)
    r = np.concatenate([r, r], axis=-1)
    bound = np.maximum(np.abs(a), np.abs(b)) * 2.0 ** -7 + r * 2.0 ** -21 + 2.0 ** -133
    return np.abs(a - b) <= bound


APPEND_CASES = [
    # name, B, Hkv, D, prefix, suffix
    ("d128_midpage", 3, 8, 128, [37, 300, 0], [129, 70, 200]),
    ("d64_aligned", 2, 2, 64, [256, 16], [64, 99]),
    ("long_positions", 2, 8, 128, [140000, 7], [40, 1]),
]


@pytest.mark.parametrize("case", APPEND_CASES, ids=[c[0] for c in APPEND_CASES])
def test_rope_append_against_oracle(rr, case):
    name, B, Hkv, D, P, S = case
    wl = synth.custom(name, B, Hkv, Hkv, D, P, S, seed=11)
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(int(max(np.add(P, S))) + 1, D, BASE)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append_rope(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    gk, gv = u16(g["k_pool"]), u16(g["v_pool"])
    assert np.array_equal(gv, vp)
    # the suffix slots: K within one unit in the last place; every other slot untouched (bit-exact)
    touched = np.zeros(kp.shape[:2], dtype=bool)
    for b in range(B):
        for j in range(S[b]):
            pos = P[b] + j
            touched[wl.page_table[b, pos // wl.ps], pos % wl.ps] = True
    assert np.array_equal(gk[~touched], kp[~touched])
    ok = _within_bound(gk[touched], kp[touched])
    assert ok.all(), f"{(~ok).sum()} rotated K elements outside the rotation's error bound"
    exact = np.mean(gk[touched] == kp[touched])
    assert exact > 0.999, f"only {exact:.5f} of the rotated K elements are bit-exact"


ATTN_CASES = [
    # name, B, Hq, Hkv, D, prefix, suffix
    ("d128_g4_midpage", 3, 8, 2, 128, [37, 300, 0], [129, 70, 200]),
    ("d128_g8", 2, 16, 2, 128, [700, 33], [90, 41]),
    ("d128_g1", 2, 2, 2, 128, [150, 0], [300, 257]),
    ("d128_g16", 1, 16, 1, 128, [77], [40]),
    ("d64_g4", 3, 8, 2, 64, [128, 999, 16], [33, 66, 130]),
    ("d64_g2_midpage", 2, 4, 2, 64, [9, 250], [129, 3]),
    ("zero_suffix_agents", 4, 8, 2, 128, [64, 300, 50, 0], [0, 70, 0, 33]),
    ("split_long_prefix", 1, 8, 2, 128, [20001], [50]),
    ("positions_past_1e5", 1, 8, 2, 128, [150000], [64]),
]


def _run_gpu_rope(rr, wl, g, table, scale=0.0):
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                              softmax_scale=scale, rope=table)
    assert rr.device_error() == 0, rr.last_error()
    return out


@pytest.mark.parametrize("case", ATTN_CASES, ids=[c[0] for c in ATTN_CASES])
def test_rope_attention_against_oracle(rr, case):
    name, B, Hq, Hkv, D, P, S = case
    wl = synth.custom(name, B, Hq, Hkv, D, P, S, seed=13)
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(int(max(np.add(P, S))) + 1, D, BASE)
    out = _run_gpu_rope(rr, wl, g, table)
    kp, vp = oracle.kv_append_rope(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    ref = oracle.extend_attention_rope(host["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens, BASE,
                                       scale=1.0 / math.sqrt(D))
    check_close(to_f64(out), ref, name)


def test_rope_changes_the_result(rr):
    """Rotation is applied: the rotated and un-rotated attention differ well beyond the parity bar."""
    wl = synth.custom("differs", 2, 8, 2, 128, [300, 40], [100, 60], seed=14)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(512, 128, BASE)
    out_r = to_f64(_run_gpu_rope(rr, wl, g, table))
    g2 = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g2["k_new"], g2["v_new"], g2["k_pool"], g2["v_pool"], g2["page_table"], g2["prefix_lens"],
                 g2["suffix_lens"])
    out_p = to_f64(rr.extend_attention(g2["q"], g2["k_pool"], g2["v_pool"], g2["page_table"], g2["prefix_lens"],
                                       g2["suffix_lens"]))
    assert np.abs(out_r - out_p).max() > 0.1


def test_rope_step_equals_its_two_calls(rr):
    wl = synth.custom("step", 3, 8, 2, 128, [37, 2000, 0], [129, 70, 300], seed=15)
    table = rr.rope_table(2100, 128, BASE)
    g1 = synth.gpu_tensors(wl, "cuda")
    out1 = _run_gpu_rope(rr, wl, g1, table)
    g2 = synth.gpu_tensors(wl, "cuda")
    out2 = rr.extend_step(g2["q"], g2["k_new"], g2["v_new"], g2["k_pool"], g2["v_pool"], g2["page_table"],
                          g2["prefix_lens"], g2["suffix_lens"], rope=table)
    assert rr.device_error() == 0, rr.last_error()
    np.testing.assert_array_equal(bf16_bits(out1), bf16_bits(out2))
    np.testing.assert_array_equal(u16(g1["k_pool"]), u16(g2["k_pool"]))
    np.testing.assert_array_equal(u16(g1["v_pool"]), u16(g2["v_pool"]))


def test_rope_position_zero_row_unrotated(rr):
    """An agent without prefix: its first token sits at position 0, so its stored K row is k_new itself."""
    wl = synth.custom("pos0", 1, 8, 2, 128, [0], [5], seed=16)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(8, 128, BASE)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    assert rr.device_error() == 0
    page = int(wl.page_table[0, 0])
    np.testing.assert_array_equal(u16(g["k_pool"][page, 0]), u16(g["k_new"][0]))


def test_rope_position_past_table_is_reported(rr):
    import torch
    wl = synth.custom("short_table", 2, 8, 2, 128, [100, 10], [20, 5], seed=17)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(110, 128, BASE)        # agent 0 reaches position 119
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    assert rr.device_error() == rr.RR_ERR_LENS
    rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                        rope=table)
    assert rr.device_error() == rr.RR_ERR_LENS
    with pytest.raises(ValueError):               # a table for another head dim
        rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                            rope=rr.rope_table(200, 64, BASE))
    with pytest.raises(rr.RRError):
        rr.rope_table(10, 96, BASE)
    # the library still works
    table = rr.rope_table(200, 128, BASE)
    g = synth.gpu_tensors(wl, "cuda")
    out = _run_gpu_rope(rr, wl, g, table)
    assert torch.isfinite(out.float()).all()


DECODE_CASES = [
    # name, B, Hq, Hkv, D, kv_lens
    ("dec_d128_g4", 4, 8, 2, 128, [300, 1000, 129, 2048]),
    ("dec_d128_g16", 2, 16, 1, 128, [900, 260]),
    ("dec_d64_g8", 2, 16, 2, 64, [555, 4096]),
    ("dec_d128_g1", 2, 2, 2, 128, [640, 33]),
    ("dec_d64_g2", 3, 4, 2, 64, [1, 17, 300]),
    ("dec_split_long", 1, 8, 2, 128, [20000]),
    ("dec_positions_past_1e5", 1, 8, 2, 128, [150001]),
]


@pytest.mark.parametrize("case", DECODE_CASES, ids=[c[0] for c in DECODE_CASES])
def test_rope_decode_against_oracle(rr, case):
    """Decode with rotary embedding: the new token's K rotated by the append, its q by the decode kernel."""
    import torch
    name, B, Hq, Hkv, D, L = case
    L = np.asarray(L, dtype=np.int64)
    wl = synth.custom(name, B, Hq, Hkv, D, L - 1, np.ones(B, dtype=np.int64), seed=19)
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(int(L.max()), D, BASE)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    out = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, rope=table)
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append_rope(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    ref = oracle.decode_attention_rope(host["q"], kp, vp, wl.page_table, L, BASE, scale=1.0 / math.sqrt(D))
    check_close(to_f64(out), ref, name)


def test_rope_decode_position_past_table_is_reported(rr):
    import torch
    wl = synth.custom("dec_short_table", 2, 8, 2, 128, [99, 10], [1, 1], seed=20)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(200, 128, BASE)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    assert rr.device_error() == 0
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, rope=rr.rope_table(50, 128, BASE))
    assert rr.device_error() == rr.RR_ERR_LENS      # agent 0's token sits at position 99
    out = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, rope=table)
    assert rr.device_error() == 0
    assert torch.isfinite(out.float()).all()

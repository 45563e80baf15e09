"""Every supported page size (8, 16, 32, 64, 128 tokens): append, extend, decode, the fused step and the
rotary-embedding calls.

The page gather issues one TMA box per page (128 / page_size lanes per 128-key tile), the append
and the fused writer index slots by position % page_size, and the last-page clearing depends on
where an agent ends inside its page; these cases exercise each size with mid-page prefixes, a
split-K batch and one-token suffixes, against the fp64 oracle (pools bit-exact).
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, to_f64

pytestmark = pytest.mark.gpu

PAGE_SIZES = [8, 32, 64, 128]


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
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def oracle_step(wl):
    h = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(h["k_new"], h["v_new"], h["k_pool"], h["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    out = oracle.extend_attention(h["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                  scale=1.0 / math.sqrt(wl.D))
    return kp, vp, out


@pytest.mark.parametrize("ps", PAGE_SIZES)
def test_extend_and_append(rr, ps):
    wl = synth.custom(f"ps{ps}", 3, 8, 2, 128, [37, 300, 0], [129, 70, 200], ps=ps, seed=3)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"])
    assert rr.device_error() == 0, rr.last_error()
    kp, vp, ref = oracle_step(wl)
    np.testing.assert_array_equal(u16(g["k_pool"]), kp)
    np.testing.assert_array_equal(u16(g["v_pool"]), vp)
    check_close(to_f64(out), ref, f"extend ps={ps}")


@pytest.mark.parametrize("ps", PAGE_SIZES)
def test_fused_step(rr, ps):
    wl = synth.custom(f"fps{ps}", 3, 8, 2, 64, [5, 250, 64], [100, 1, 77], ps=ps, seed=3)
    g = synth.gpu_tensors(wl, "cuda")
    out_f = rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                           g["prefix_lens"], g["suffix_lens"])
    assert rr.device_error() == 0, rr.last_error()
    kp, vp, ref = oracle_step(wl)
    np.testing.assert_array_equal(u16(g["k_pool"]), kp)
    np.testing.assert_array_equal(u16(g["v_pool"]), vp)
    check_close(to_f64(out_f), ref, f"fused ps={ps}")
    g2 = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g2["k_new"], g2["v_new"], g2["k_pool"], g2["v_pool"], g2["page_table"], g2["prefix_lens"],
                 g2["suffix_lens"])
    out_u = rr.extend_attention(g2["q"], g2["k_pool"], g2["v_pool"], g2["page_table"], g2["prefix_lens"],
                                g2["suffix_lens"])
    np.testing.assert_array_equal(bf16_bits(out_f), bf16_bits(out_u))


@pytest.mark.parametrize("ps", PAGE_SIZES)
def test_decode(rr, ps):
    import torch
    L = np.array([1, 2 * ps + 3, 1000, 129], dtype=np.int64)
    wl = synth.custom(f"dps{ps}", 4, 16, 2, 128, L - 1, np.ones(4, dtype=np.int64), ps=ps, seed=3)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], (g["prefix_lens"] + 1).to(torch.int32))
    assert rr.device_error() == 0, rr.last_error()
    kp, vp, ref = oracle_step(wl)
    check_close(to_f64(out), ref, f"decode ps={ps}")


@pytest.mark.parametrize("ps", [8, 128])
def test_split_k(rr, ps):
    wl = synth.custom(f"sps{ps}", 1, 8, 2, 128, [9000 + 5], [60], ps=ps, seed=3)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"])
    assert rr.device_error() == 0, rr.last_error()
    _, _, ref = oracle_step(wl)
    check_close(to_f64(out), ref, f"split ps={ps}")


@pytest.mark.parametrize("ps", PAGE_SIZES)
def test_rotary_extend_and_decode(rr, ps):
    """Rotary embedding at every page size: the rotated append indexes slots by position % page_size."""
    import torch
    base = 500000.0
    wl = synth.custom(f"rope_ps{ps}", 3, 8, 2, 128, [37, 300, 0], [129, 70, 200], ps=ps, seed=4)
    h = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    table = rr.rope_table(600, 128, base)
    out = rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                         g["prefix_lens"], g["suffix_lens"], rope=table)
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append_rope(h["k_new"], h["v_new"], h["k_pool"], h["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, base)
    np.testing.assert_array_equal(u16(g["v_pool"]), vp)
    ref = oracle.extend_attention_rope(h["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens, base,
                                       scale=1.0 / math.sqrt(wl.D))
    check_close(to_f64(out), ref, f"rotary extend ps={ps}")
    # decode over one new token per agent at its next position
    L = np.array([400, 77, 513], dtype=np.int64)
    wd = synth.custom(f"rope_dec_ps{ps}", 3, 8, 2, 128, L - 1, np.ones(3, dtype=np.int64), ps=ps, seed=5)
    hd = synth.cpu_tensors(wd)
    gd = synth.gpu_tensors(wd, "cuda")
    rr.kv_append(gd["k_new"], gd["v_new"], gd["k_pool"], gd["v_pool"], gd["page_table"], gd["prefix_lens"],
                 gd["suffix_lens"], rope=table)
    kv = (gd["prefix_lens"] + 1).to(torch.int32)
    outd = rr.decode_attention(gd["q"], gd["k_pool"], gd["v_pool"], gd["page_table"], kv, rope=table)
    assert rr.device_error() == 0, rr.last_error()
    kpd, vpd = oracle.kv_append_rope(hd["k_new"], hd["v_new"], hd["k_pool"], hd["v_pool"], wd.page_table,
                                     wd.prefix_lens, wd.suffix_lens, base)
    refd = oracle.decode_attention_rope(hd["q"], kpd, vpd, wd.page_table, L, base, scale=1.0 / math.sqrt(wd.D))
    check_close(to_f64(outd), refd, f"rotary decode ps={ps}")

"""The rr_tensor calls on the GPU: on contiguous tensors they give bit for bit what the plain calls give (and
so match the oracle); views the kernels cannot take are rejected by the library before any launch."""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def test_tensor_calls_match_plain_calls_and_oracle(rr):
    import torch
    wl = synth.custom("tensors", 3, 8, 2, 128, [300, 0, 77], [70, 150, 33], seed=4)
    a = synth.gpu_tensors(wl, "cuda")
    b = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(a["k_new"], a["v_new"], a["k_pool"], a["v_pool"], a["page_table"], a["prefix_lens"],
                 a["suffix_lens"])
    out_a = rr.extend_attention(a["q"], a["k_pool"], a["v_pool"], a["page_table"], a["prefix_lens"],
                                a["suffix_lens"])
    rr.kv_append_tensors(b["k_new"], b["v_new"], b["k_pool"], b["v_pool"], b["page_table"], b["prefix_lens"],
                         b["suffix_lens"])
    out_b = torch.empty_like(b["q"])
    rr.extend_attention_tensors(b["q"], b["k_pool"], b["v_pool"], b["page_table"], b["prefix_lens"],
                                b["suffix_lens"], out_b)
    assert rr.device_error() == 0, rr.last_error()
    for k in ("k_pool", "v_pool"):
        np.testing.assert_array_equal(bf16_bits(a[k]), bf16_bits(b[k]))
    np.testing.assert_array_equal(bf16_bits(out_a), bf16_bits(out_b))
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    np.testing.assert_array_equal(bf16_bits(b["k_pool"]), kp)
    ref = oracle.extend_attention(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                  scale=1.0 / math.sqrt(wl.D))
    check_close(to_f64(out_b), ref, "tensor calls")


def test_views_the_kernels_cannot_take_are_rejected(rr):
    import torch
    wl = synth.custom("views", 2, 8, 2, 128, [64, 16], [20, 12], seed=5)
    g = synth.gpu_tensors(wl, "cuda")
    out = torch.full_like(g["q"], 7.0)
    wide = torch.zeros((wl.T, wl.Hq, 2 * wl.D), dtype=torch.bfloat16, device="cuda")
    wide[:, :, :wl.D] = g["q"]
    strided_q = wide[:, :, :wl.D]                 # rows 512 elements apart instead of 128
    args = (g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    with pytest.raises(rr.RRError) as e:
        rr.extend_attention_tensors(strided_q, *args, out)
    assert e.value.code == rr.RR_ERR_UNSUPPORTED and "stride" in str(e.value)
    with pytest.raises(rr.RRError) as e:
        rr.extend_attention_tensors(g["q"], g["k_pool"], g["v_pool"], g["page_table"],
                                    g["prefix_lens"].to(torch.int64), g["suffix_lens"], out)
    assert e.value.code == rr.RR_ERR_UNSUPPORTED and "prefix_lens" in str(e.value)
    with pytest.raises(rr.RRError) as e:
        rr.kv_append_tensors(g["k_new"], g["v_new"], g["k_pool"].transpose(1, 2), g["v_pool"], g["page_table"],
                             g["prefix_lens"], g["suffix_lens"])
    assert e.value.code in (rr.RR_ERR_UNSUPPORTED, rr.RR_ERR_INVALID_ARG)
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())               # nothing was launched
    assert rr.device_error() == 0

"""Decode attention (one new token per agent) on the GPU vs the fp64 oracle, element by element.

Cases span every head dim and GQA group, key counts below, at and just past tile (128) and page
(16) boundaries, single-key agents, split-K batches (few agents, long contexts), shared prefix
pages, and the three full-size decode batches on sampled agents.  Pool slots no agent owns hold
NaN, so reading one poisons the output.  The decode kernel is also checked against the extend
path on the same inputs, for page-placement bit-exactness, and for its error reporting.
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, oracle_sampled, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def decode_workload(name, B, Hq, Hkv, D, L, shared=0, seed=17, num_pages=None):
    L = np.asarray(L, dtype=np.int64)
    return synth.custom(name, B, Hq, Hkv, D, L - 1, np.ones(B, dtype=np.int64), shared_len=shared, seed=seed,
                        num_pages=num_pages)


def run_decode(rr, wl, g=None, scale=0.0):
    import torch
    g = g if g is not None else synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    out = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, softmax_scale=scale)
    assert rr.device_error() == 0, rr.last_error()
    return out, g


def oracle_decode(wl, scale=None):
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    L = (np.asarray(wl.prefix_lens) + 1).astype(np.int32)
    return oracle.decode_attention(t["q"], kp, vp, wl.page_table, L, scale=scale)


CASES = [
    # name, B, Hq, Hkv, D, kv_lens
    ("d128_g4_mixed", 4, 8, 2, 128, [300, 1000, 129, 2048]),
    ("d128_g8", 3, 16, 2, 128, [511, 77, 1500]),
    ("d128_g1", 2, 2, 2, 128, [640, 33]),
    ("d128_g2", 2, 4, 2, 128, [700, 1100]),
    ("d128_g16", 2, 16, 1, 128, [900, 260]),
    ("d64_g4", 3, 8, 2, 64, [129, 1023, 2000]),
    ("d64_g8", 2, 16, 2, 64, [555, 4096]),
    ("single_key_agents", 3, 8, 2, 128, [1, 1, 2]),
    ("tile_boundaries", 5, 8, 2, 128, [127, 128, 129, 255, 256]),
    ("page_boundaries", 4, 8, 2, 128, [15, 16, 17, 33]),
    ("split_one_long_agent", 1, 8, 2, 128, [20000]),
    ("split_two_agents_d64", 2, 8, 2, 64, [9000, 3100]),
    ("split_g8_midpage", 1, 16, 2, 128, [12345]),
    # every agent's last page partly its own, on tiles 0-7 of the agent and split into pieces of different
    # lengths: a CTA's producer warps take its tiles in turn, so the tail tiles fall to both producers and
    # both side barriers that hold a partly owned V page are used in one call
    ("tails_alternate_producers", 8, 8, 2, 128, [128 * k + 5 + 2 * k for k in range(8)]),
    ("tails_alternate_producers_d64", 7, 8, 2, 64, [128 * k + 9 for k in range(7)]),
    ("tails_split_one_agent", 1, 8, 2, 128, [9 * 1024 + 7]),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_decode_matches_oracle(rr, case):
    name, B, Hq, Hkv, D, L = case
    wl = decode_workload(name, B, Hq, Hkv, D, L)
    out, _ = run_decode(rr, wl)
    check_close(to_f64(out), oracle_decode(wl, 1.0 / math.sqrt(D)), name)


def test_decode_shared_prefix_pages(rr):
    # every agent's first 64 positions live on the same physical pages (read by all, written by none)
    wl = decode_workload("shared", 4, 8, 2, 128, [64 + 1, 300, 1000, 129], shared=64)
    out, _ = run_decode(rr, wl)
    check_close(to_f64(out), oracle_decode(wl, 1.0 / math.sqrt(128)), "shared")


def test_decode_explicit_scale(rr):
    wl = decode_workload("scale", 2, 8, 2, 128, [400, 900])
    out, _ = run_decode(rr, wl, scale=0.05)
    check_close(to_f64(out), oracle_decode(wl, 0.05), "scale")


def test_decode_single_key_is_value_exactly(rr):
    import torch
    wl = decode_workload("one", 3, 8, 2, 128, [1, 1, 1])
    out, g = run_decode(rr, wl)
    v = g["v_new"].float()                                    # [B, Hkv, D]
    ref = v.repeat_interleave(4, dim=1)                       # head h reads KV head h // G
    assert torch.equal(out.float(), ref)


def test_decode_equals_extend_path(rr):
    """The same batch through rr_extend_attention with suffix 1: both within the parity bar of each other."""
    wl = decode_workload("vs_extend", 4, 8, 2, 128, [5000, 129, 2047, 64])
    out, g = run_decode(rr, wl)
    ext = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    assert rr.device_error() == 0
    check_close(to_f64(out), to_f64(ext), "decode vs extend")


def test_decode_page_permutation_bit_exact(rr):
    a = decode_workload("pa", 3, 8, 2, 128, [3000, 700, 129], num_pages=600)
    b = decode_workload("pb", 3, 8, 2, 128, [3000, 700, 129], num_pages=900)
    assert not np.array_equal(a.page_table, b.page_table)
    np.testing.assert_array_equal(bf16_bits(run_decode(rr, a)[0]), bf16_bits(run_decode(rr, b)[0]))


def test_decode_repeatable(rr):
    wl = decode_workload("rep", 2, 8, 2, 128, [7000, 300])
    g = synth.gpu_tensors(wl, "cuda")
    o1, _ = run_decode(rr, wl, g)
    import torch
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    o2 = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens)
    np.testing.assert_array_equal(bf16_bits(o1), bf16_bits(o2))


@pytest.mark.parametrize("name", synth.DECODE_CONFIGS)
def test_decode_full_size_configs_sampled(rr, name):
    """The full decode batch on the GPU; the oracle on every head of sampled agents' rows."""
    import torch
    free = torch.cuda.mem_get_info()[0] if name == "c4_decode" else None
    wl = synth.decode_config(name, free_hbm_bytes=free)
    out, g = run_decode(rr, wl)
    del g
    torch.cuda.empty_cache()
    got = to_f64(out)
    rng = np.random.default_rng(1)
    n_extra = 1 if name == "c4_decode" else 4  # regenerating a c4 agent's ~260k keys on the CPU is the cost
    agents = sorted(set([int(np.argmax(wl.prefix_lens)), int(np.argmin(wl.prefix_lens))]) |
                    set(int(x) for x in rng.choice(wl.B, size=n_extra, replace=False)))
    rows = {b: np.array([0], dtype=np.int64) for b in agents}
    ref = oracle_sampled(wl, rows)
    for b in agents:
        check_close(got[wl.cu[b]:wl.cu[b] + 1], ref[b], f"{name} agent {b}")
    assert np.isfinite(got).all()


def test_decode_rejects_bad_arguments(rr):
    import torch
    wl = decode_workload("bad", 2, 8, 2, 128, [100, 200])
    g = synth.gpu_tensors(wl, "cuda")
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    with pytest.raises(ValueError):  # batch of q and kv_lens disagree
        rr.decode_attention(g["q"][:1], g["k_pool"], g["v_pool"], g["page_table"], kv_lens)
    # a zero-length agent is reported on the device, and nothing is computed for the batch
    bad = kv_lens.clone()
    bad[1] = 0
    rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], bad)
    assert rr.device_error() == rr.RR_ERR_LENS
    # a page id outside the pool is reported
    pt = g["page_table"].clone()
    pt[0, 0] = wl.num_pages + 5
    rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], pt, kv_lens)
    assert rr.device_error() == rr.RR_ERR_OOB
    # and the library still works afterwards
    out, _ = run_decode(rr, wl)
    assert np.isfinite(to_f64(out)).all()


@pytest.mark.parametrize("L", [[2, 3, 4, 5], [130, 20000]], ids=["few_keys", "split"])
def test_decode_unit_values_give_unit_output(rr, L):
    """V == 1: the weight sum and the P^T operand hold the same bf16-rounded weights, so every output is 1 up
    to fp32 summation order, which rounds to exactly 1.0 in bf16 (the second batch splits its key range and
    goes through the combine)."""
    wl = decode_workload("ones", len(L), 8, 2, 128, L)
    g = synth.gpu_tensors(wl, "cuda")
    g["v_new"].fill_(1.0)
    for b in range(wl.B):
        for lp in range(-(-int(wl.prefix_lens[b]) // wl.ps)):
            g["v_pool"][int(wl.page_table[b, lp])] = 1.0
    out, _ = run_decode(rr, wl, g=g)
    np.testing.assert_array_equal(to_f64(out), 1.0)

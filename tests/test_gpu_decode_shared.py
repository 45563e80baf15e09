"""Decode over a shared prefix (rr_decode_attention_shared) on the GPU against the fp64 oracle.

Every agent's first shared_len positions are the same physical pages (a common system prompt).  The
call reads them once per group of 16 / G agents and merges each (agent, head)'s shared and private
partial results; the oracle is the plain decode definition over each agent's whole key range.  Cases:
every GQA group (groups of 16, 8, 4, 2 and 1 agents), both head dims, batches that leave the last group
partly empty, a batch small enough for the private part to be split, a c5-shaped batch, and the errors
the schedule reports (a page table that leaves the shared prefix, an agent with no private key).
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import check_close, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def workload(name, B, Hq, Hkv, D, shared, L, seed=23, ps=16):
    L = np.asarray(L, dtype=np.int64)
    return synth.custom(name, B, Hq, Hkv, D, L - 1, np.ones(B, dtype=np.int64), shared_len=shared, seed=seed, ps=ps)


def run(rr, wl, shared):
    import torch
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    kv = (g["prefix_lens"] + 1).to(torch.int32)
    out = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv, shared_len=shared)
    return out, g, kv


def reference(wl):
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    L = (np.asarray(wl.prefix_lens) + 1).astype(np.int32)
    return oracle.decode_attention(t["q"], kp, vp, wl.page_table, L, scale=1.0 / math.sqrt(wl.D))


rng = np.random.default_rng(5)
CASES = [
    # name, B, Hq, Hkv, D, shared_len, kv_lens
    ("g4_d128_partial_group", 6, 8, 2, 128, 256, [300, 1000, 257, 2048, 700, 400]),
    ("g8_d128", 5, 16, 2, 128, 512, [600, 513, 2000, 900, 1500]),
    ("g1_d128", 20, 2, 2, 128, 128, list(rng.integers(129, 1500, 20))),
    ("g2_d64", 9, 4, 2, 64, 384, list(rng.integers(385, 3000, 9))),
    ("g16_d128", 3, 16, 1, 128, 256, [400, 300, 900]),
    ("g4_d64_ps64", 7, 8, 2, 64, 640, list(rng.integers(641, 2500, 7))),
    ("split_private_part", 2, 8, 2, 128, 4096, [20000, 9000]),
    ("c5_shaped", 64, 32, 8, 128, 4096, list(4096 + rng.integers(4096, 16384, 64))),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_shared_prefix_decode_matches_oracle(rr, case):
    name, B, Hq, Hkv, D, shared, L = case
    wl = workload(name, B, Hq, Hkv, D, shared, L, ps=64 if "ps64" in name else 16)
    out, _, _ = run(rr, wl, shared)
    assert rr.device_error() == 0, rr.last_error()
    check_close(to_f64(out), reference(wl), name)


def test_shared_prefix_decode_agrees_with_plain_decode(rr):
    wl = workload("vs_plain", 12, 32, 8, 128, 1024, list(rng.integers(1025, 6000, 12)))
    out, g, kv = run(rr, wl, 1024)
    plain = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv)
    assert rr.device_error() == 0
    check_close(to_f64(out), to_f64(plain), "shared vs plain")


def test_shared_prefix_decode_errors(rr):
    import torch
    wl = workload("errs", 5, 8, 2, 128, 256, [400, 300, 900, 700, 260])
    out, g, kv = run(rr, wl, 256)
    assert rr.device_error() == 0
    with pytest.raises(rr.RRError):           # not a multiple of 128
        rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv, shared_len=200)
    # an agent whose keys end inside the shared prefix
    short = kv.clone()
    short[2] = 256
    rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], short, shared_len=256)
    assert rr.device_error() == rr.RR_ERR_LENS
    # an agent whose page table leaves the shared prefix
    pt = g["page_table"].clone()
    pt[3, 1] = pt[3, 1] + 1
    rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], pt, kv, shared_len=256)
    assert rr.device_error() == rr.RR_ERR_SHARED
    # the library still works
    out2 = rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv, shared_len=256)
    assert rr.device_error() == 0
    assert torch.equal(out2, out)

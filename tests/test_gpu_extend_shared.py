"""rr_extend_attention_shared: extend attention over a prefix every agent shares, as a cascade (a pass of
every suffix row against the shared keys in dense Q tiles that cross agents, then each agent's own keys,
merged by log-sum-exp weights), against the fp64 oracle element by element and against the plain call.

Cases span every head dim and GQA group, agents whose prefix is exactly the shared part, mid-page
prefixes, batches whose suffixes are short enough that one dense tile holds rows of several agents, and
the full-size shared-prefix batch (sampled rows); the device-side checks (a page table that leaves the
shared pages, a prefix shorter than the shared part) report their codes and write nothing.
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, oracle_sampled, sample_rows, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def appended(rr, wl):
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    return g


def run_oracle(wl):
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    return oracle.extend_attention(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                   scale=1.0 / math.sqrt(wl.D))


CASES = [
    # name, B, Hq, Hkv, D, shared_len, prefix, suffix
    ("d128_g4", 3, 8, 2, 128, 128, [165, 256, 640], [70, 1, 200]),
    ("d128_g8_prefix_is_shared", 3, 16, 2, 128, 256, [256, 300, 256], [40, 129, 7]),
    ("d128_g1", 2, 2, 2, 128, 128, [128, 700], [130, 64]),
    ("d128_g2", 2, 4, 2, 128, 384, [400, 384], [33, 90]),
    ("d128_g16", 2, 16, 1, 128, 128, [129, 500], [20, 11]),
    ("d64_g4", 3, 8, 2, 64, 128, [200, 128, 1000], [45, 100, 3]),
    ("tiles_cross_agents", 9, 8, 2, 128, 256, [256, 270, 300, 512, 256, 777, 260, 256, 400],
     [5, 17, 40, 3, 29, 1, 12, 33, 8]),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_shared_cascade_matches_oracle_and_plain_call(rr, case):
    name, B, Hq, Hkv, D, shared, P, S = case
    wl = synth.custom(name, B, Hq, Hkv, D, P, S, shared_len=shared, seed=7)
    g = appended(rr, wl)
    args = (g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    out = rr.extend_attention(*args, shared_len=shared)
    plain = rr.extend_attention(*args)
    assert rr.device_error() == 0, rr.last_error()
    ref = run_oracle(wl)
    got = to_f64(out)
    check_close(got, ref, f"shared {name}")
    check_close(got, to_f64(plain), f"shared {name} vs rr_extend_attention")


def test_shared_pages_must_match(rr):
    import torch
    wl = synth.custom("mismatch", 3, 8, 2, 128, [256, 300, 400], [20, 30, 40], shared_len=256, seed=8)
    g = appended(rr, wl)
    pt = g["page_table"].clone()
    pt[2, 3] = int(wl.page_table[2, 20])  # agent 2's fourth shared page replaced by one of its private pages
    out = torch.full_like(g["q"], 3.0)
    rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], pt, g["prefix_lens"], g["suffix_lens"], out=out,
                        shared_len=256)
    assert rr.device_error() == rr.RR_ERR_SHARED
    assert bool((out == 3.0).all())


def test_prefix_shorter_than_shared_part_is_rejected(rr):
    import torch
    # the shared pages do match (agent 1's first 8 pages are agent 0's): only its prefix is too short
    wl = synth.custom("short", 2, 8, 2, 128, [256, 100], [20, 30], shared_len=128, seed=9)
    g = appended(rr, wl)
    out = torch.full_like(g["q"], 3.0)
    rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                        out=out, shared_len=128)
    assert rr.device_error() == rr.RR_ERR_LENS
    assert bool((out == 3.0).all())


def test_host_side_arguments(rr):
    wl = synth.custom("args", 2, 8, 2, 128, [256, 300], [20, 30], shared_len=128, seed=10)
    g = appended(rr, wl)
    args = (g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    for bad in (64, 200, -128):
        with pytest.raises(rr.RRError) as e:
            rr.extend_attention(*args, shared_len=bad)
        assert e.value.code == rr.RR_ERR_UNSUPPORTED
    with pytest.raises(rr.RRError) as e:
        rr.extend_attention(*args, shared_len=128 * 1000)
    assert e.value.code == rr.RR_ERR_INVALID_ARG


def test_full_size_shared_prefix_batch(rr):
    """c5_shared (128 agents over a 4096-token common prefix): sampled rows against the oracle, every row
    against the plain call."""
    import torch
    wl = synth.config("c5_shared")
    g = appended(rr, wl)
    args = (g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    out = rr.extend_attention(*args, shared_len=wl.shared_len)
    plain = rr.extend_attention(*args)
    assert rr.device_error() == 0, rr.last_error()
    check_close(to_f64(out), to_f64(plain), "c5_shared cascade vs rr_extend_attention (all rows)")
    rows = sample_rows(wl, flop_budget=1.5e11, seed=3, max_agents=8)
    ref = oracle_sampled(wl, rows, 1.0 / math.sqrt(wl.D))
    got_rows, ref_rows = [], []
    for b, rs in rows.items():
        got_rows.append(to_f64(out[torch.from_numpy(wl.cu[b] + rs).cuda()]))
        ref_rows.append(ref[b])
    check_close(np.concatenate(got_rows), np.concatenate(ref_rows), "c5_shared cascade vs oracle")
    del g, out, plain
    torch.cuda.empty_cache()

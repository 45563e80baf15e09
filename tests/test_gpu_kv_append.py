"""KV append on the GPU vs the oracle: bit-exact on every pool byte; bad inputs become device errors."""
import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def _run(rr, wl, pool_fill=0x1357):
    g = synth.gpu_tensors(wl, "cuda", pool_fill=pool_fill)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    code = rr.device_error()
    return g, code


def _expected(wl, pool_fill=0x1357):
    t = synth.cpu_tensors(wl, pool_fill=pool_fill)
    return oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                            wl.suffix_lens)


SMALL = [
    ("d64_g4", 3, 8, 2, 64, [48, 0, 35], [17, 40, 1]),
    ("d128_midpage", 4, 32, 8, 128, [100, 7, 0, 256], [29, 200, 16, 0]),
    ("d128_one_token", 1, 4, 4, 128, [15], [1]),
]


@pytest.mark.parametrize("case", SMALL, ids=[c[0] for c in SMALL])
def test_append_bit_exact_small(rr, case):
    name, B, Hq, Hkv, D, P, S = case
    wl = synth.custom(name, B, Hq, Hkv, D, P, S, seed=4)
    g, code = _run(rr, wl)
    assert code == 0
    kp, vp = _expected(wl)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)


@pytest.mark.parametrize("name", ["c1_tiny", "c5_shared"])
def test_append_bit_exact_config(rr, name):
    wl = synth.config(name)
    g, code = _run(rr, wl)
    assert code == 0
    kp, vp = _expected(wl)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)   # every byte of the pool, incl. sentinels
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)


def test_append_c3_rr_mid_page(rr):
    # histories minus equal tail chunks: every append starts mid-page
    wl = synth.config("c3_rr")
    assert np.any(wl.prefix_lens % wl.ps != 0)
    g, code = _run(rr, wl)
    assert code == 0
    kp, vp = _expected(wl)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)


def test_append_empty_batch_and_zero_suffix(rr):
    wl = synth.custom("z", 2, 4, 2, 64, [32, 16], [0, 0], seed=1)
    g, code = _run(rr, wl)
    assert code == 0
    kp, vp = _expected(wl)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)


def test_append_bad_page_is_a_device_error(rr):
    import torch
    wl = synth.custom("bad", 2, 4, 2, 64, [16, 0], [10, 20], seed=2)
    g = synth.gpu_tensors(wl, "cuda", pool_fill=0x1357)
    before = bf16_bits(g["k_pool"]).copy()
    pt = g["page_table"].clone()
    pt[1, 0] = wl.num_pages + 5
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], pt, g["prefix_lens"], g["suffix_lens"])
    assert rr.device_error() == rr.RR_ERR_OOB
    after = bf16_bits(g["k_pool"])
    # agent 0 and agent 1's second page written; agent 1's first page (now out of range) skipped
    kp, _ = _expected(wl)
    skipped = int(wl.page_table[1, 0])
    kp[skipped] = before[skipped]
    np.testing.assert_array_equal(after, kp)
    assert rr.device_error() == 0   # the word was cleared by the previous read
    del torch


def test_append_lens_mismatch_is_a_device_error(rr):
    wl = synth.custom("lm", 2, 4, 2, 64, [16, 0], [10, 20], seed=2)
    g = synth.gpu_tensors(wl, "cuda", pool_fill=0x1357)
    before = bf16_bits(g["k_pool"]).copy()
    sl = g["suffix_lens"].clone()
    sl[1] = 21                      # sum no longer equals the rows of k_new
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], sl)
    assert rr.device_error() == rr.RR_ERR_LENS
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), before)   # nothing written


def test_append_rejects_bad_arguments(rr):
    import torch
    wl = synth.custom("a", 1, 4, 2, 64, [0], [4], seed=2)
    g = synth.gpu_tensors(wl, "cuda")
    with pytest.raises(TypeError):
        rr.kv_append(g["k_new"].float(), g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])
    with pytest.raises(ValueError):
        rr.kv_append(g["k_new"][:, :1], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])
    del torch


@pytest.mark.parametrize("B", [2047, 2048, 3001])
def test_append_bit_exact_many_agents(rr, B):
    """Up to 2047 agents the append kernel checks and sums the lengths itself; beyond, the schedule kernel does it
    first.  Both sides of the switch, mid-page prefixes and empty suffixes among them, land bit-exact."""
    rng = np.random.default_rng(B)
    P = rng.integers(0, 40, size=B)
    S = rng.integers(0, 4, size=B)
    wl = synth.custom(f"many_{B}", B, 4, 2, 64, P, S, seed=9)
    g, code = _run(rr, wl)
    assert code == 0
    kp, vp = _expected(wl)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)


@pytest.mark.parametrize("B", [2, 2100])
def test_append_negative_prefix_is_a_device_error(rr, B):
    """A negative cached length fails the check on either path: RR_ERR_LENS, nothing written."""
    P = np.full(B, 16, dtype=np.int64)
    S = np.full(B, 2, dtype=np.int64)
    wl = synth.custom(f"negp_{B}", B, 4, 2, 64, P, S, seed=3)
    g = synth.gpu_tensors(wl, "cuda", pool_fill=0x1357)
    before = bf16_bits(g["k_pool"]).copy()
    pl = g["prefix_lens"].clone()
    pl[B - 1] = -1
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], pl, g["suffix_lens"])
    assert rr.device_error() == rr.RR_ERR_LENS
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), before)

"""Split-K path: batches with fewer work units than two waves of SMs split every unit's key range,
compute partial (max, sum, unnormalised output) per piece and merge them by log-sum-exp.

Checked element by element against the fp64 oracle, for both head dims, plus page-permutation
bit-exactness (the split decision depends only on the lengths) and the device-side item count
(the split really happened)."""
import ctypes
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


def run(rr, wl, g=None):
    g = g if g is not None else synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"])
    assert rr.device_error() == 0, rr.last_error()
    return out


def ref(wl):
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    return oracle.extend_attention(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                   scale=1 / math.sqrt(wl.D))


CASES = [
    # a single returning agent with a long surviving prefix: two units for 150 SMs
    ("one_agent_long_prefix", 1, 8, 2, 128, [20000], [50]),
    ("one_agent_g8", 1, 16, 2, 128, [9000], [130]),
    ("two_agents_d64", 2, 8, 2, 64, [12000, 3000], [70, 200]),
    ("mid_page_tail", 1, 4, 1, 128, [7777], [33]),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_split_matches_oracle(rr, case):
    name, B, Hq, Hkv, D, P, S = case
    wl = synth.custom(name, B, Hq, Hkv, D, P, S, seed=11)
    out = run(rr, wl)
    check_close(to_f64(out), ref(wl), name)


def test_split_happened(rr):
    import torch
    wl = synth.custom("s", 1, 8, 2, 128, [20000], [50], seed=1)
    run(rr, wl)
    torch.cuda.synchronize()
    # the workspace header holds (items, lens ok, split units): read it through a tiny device copy is not exposed,
    # so compare against the allocation-free entry point, which never splits: outputs agree within tolerance but
    # are not bit-identical (different summation order), which shows the split path ran
    fn = rr.lib().rr_extend_attention_noalloc
    fn.restype = ctypes.c_int
    fn.argtypes = [ctypes.c_void_p] * 7 + [ctypes.POINTER(rr.Dims), ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p]
    g = synth.gpu_tensors(wl, "cuda")
    split_out = run(rr, wl, g)
    plain = torch.empty_like(g["q"])
    dims = rr.make_dims(wl.B, wl.Hq, wl.Hkv, wl.D, wl.ps, wl.max_pages, wl.num_pages, wl.T)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert fn(g["q"].data_ptr(), g["k_pool"].data_ptr(), g["v_pool"].data_ptr(), g["page_table"].data_ptr(),
              g["prefix_lens"].data_ptr(), g["suffix_lens"].data_ptr(), plain.data_ptr(), ctypes.byref(dims), 0.0,
              err.data_ptr(), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)) == 0
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error {int(err.item())} in the allocation-free call"
    a, b = to_f64(split_out), to_f64(plain)
    assert np.abs(a - b).max() <= 2e-2
    assert not np.array_equal(bf16_bits(split_out), bf16_bits(plain))


def test_split_page_permutation_bit_exact(rr):
    a = synth.custom("pa", 2, 8, 2, 128, [15000, 4000], [60, 90], seed=3, num_pages=3000)
    b = synth.custom("pb", 2, 8, 2, 128, [15000, 4000], [60, 90], seed=3, num_pages=4100)
    assert not np.array_equal(a.page_table, b.page_table)
    np.testing.assert_array_equal(bf16_bits(run(rr, a)), bf16_bits(run(rr, b)))

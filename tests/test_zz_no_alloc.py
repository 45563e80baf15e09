"""rr_extend_attention_noalloc: the allocation-free variant of extend attention.

Some callers cannot allocate device memory during a call -- their memory is
wholly owned by their own pool allocator, or they cannot afford the device
synchronisation that cudaMalloc/cudaFree implies -- so this entry point keeps
its schedule scratch in a fixed static device array instead.  These tests call
it through the C ABI twice in a row (the second call reuses the array the first
one left behind) and check both outputs against the fp64 oracle (the parity
bar) and against the allocating entry point (within the same bar), on a small
ragged batch and on a batch at the 4096-agent limit; and that batches beyond
either limit of the array are rejected before anything is launched.  They live
in their own file so that they are collected after every other test.
"""
import ctypes
import math

import numpy as np
import pytest

import oracle
import synth
from parity import check_close, to_f64

pytestmark = pytest.mark.gpu


def _noalloc_fn(rr):
    fn = rr.lib().rr_extend_attention_noalloc
    vp = ctypes.c_void_p
    fn.restype = ctypes.c_int
    fn.argtypes = [vp, vp, vp, vp, vp, vp, vp, ctypes.POINTER(rr.Dims), ctypes.c_float, vp, vp]
    return fn


def _two_calls_against_oracle_and_allocating_call(wl):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as rr
    fn = _noalloc_fn(rr)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    alloc = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                g["suffix_lens"])
    assert rr.device_error() == 0
    alloc64 = to_f64(alloc)
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    ref = oracle.extend_attention(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                  scale=1.0 / math.sqrt(wl.D))
    dims = rr.make_dims(wl.B, wl.Hq, wl.Hkv, wl.D, wl.ps, wl.max_pages, wl.num_pages, wl.T)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        out = torch.full_like(g["q"], float("nan"))
        rc = fn(g["q"].data_ptr(), g["k_pool"].data_ptr(), g["v_pool"].data_ptr(), g["page_table"].data_ptr(),
                g["prefix_lens"].data_ptr(), g["suffix_lens"].data_ptr(), out.data_ptr(), ctypes.byref(dims), 0.0,
                err.data_ptr(), stream)
        assert rc == 0, rr.last_error()
        torch.cuda.synchronize()
        assert int(err.item()) == 0, f"call {call}: device error {int(err.item())}"
        got = to_f64(out)
        check_close(got, ref, f"{wl.name} call {call} vs oracle")
        check_close(got, alloc64, f"{wl.name} call {call} vs rr_extend_attention")


def test_noalloc_matches_oracle_and_allocating_entry_point_on_two_calls():
    # several agents, ragged Q tiles, a mid-page prefix and a prefix-less agent
    wl = synth.custom("noalloc", 4, 8, 2, 128, [300, 0, 1037, 64], [70, 150, 33, 257], seed=6)
    _two_calls_against_oracle_and_allocating_call(wl)


def test_noalloc_at_the_agent_limit():
    """4096 agents, the array's limit (the schedule then keeps its per-agent unit offsets in the array rather
    than in shared memory): one to three suffix tokens each over short prefixes."""
    rng = np.random.default_rng(8)
    B = 4096
    wl = synth.custom("noalloc_4096", B, 8, 2, 64, rng.integers(0, 40, B), rng.integers(1, 4, B), seed=8)
    _two_calls_against_oracle_and_allocating_call(wl)


def test_noalloc_rejects_batches_beyond_its_scratch():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as rr
    fn = _noalloc_fn(rr)
    dims = rr.make_dims(5000, 8, 2, 128, 16, 1, 1, 5000)
    x = torch.zeros(16, dtype=torch.int32, device="cuda")
    rc = fn(x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(),
            ctypes.byref(dims), 0.0, None, None)
    assert rc == rr.RR_ERR_UNSUPPORTED
    assert "static scratch" in rr.last_error()


def test_noalloc_rejects_batches_beyond_its_work_units():
    """A small batch with so many suffix tokens that its work units could exceed the array's 65536."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as rr
    fn = _noalloc_fn(rr)
    dims = rr.make_dims(2, 32, 8, 128, 16, 1, 1, 600000)  # 8 x (600000 / 64 + 3) = 75024 units
    x = torch.zeros(16, dtype=torch.int32, device="cuda")
    rc = fn(x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(), x.data_ptr(),
            ctypes.byref(dims), 0.0, None, None)
    assert rc == rr.RR_ERR_UNSUPPORTED
    assert "work units" in rr.last_error()

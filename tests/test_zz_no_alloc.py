"""rr_extend_attention_noalloc: the allocation-free variant of extend attention.

Some callers cannot allocate device memory during a call -- their memory is
wholly owned by their own pool allocator, or they cannot afford the device
synchronisation that cudaMalloc/cudaFree implies -- so this entry point keeps
its schedule scratch in a fixed static device array instead.  This test calls
it through the C ABI twice in a row (the second call reuses the array the first
one left behind) and checks both outputs against the allocating entry point
within the attention parity tolerance.  It lives in its own file so that it is
collected after every other test.
"""
import ctypes

import numpy as np
import pytest

import synth
from parity import MAX_ABS, MEAN_ABS, to_f64

pytestmark = pytest.mark.gpu


def _noalloc_fn(rr):
    fn = rr.lib().rr_extend_attention_noalloc
    vp = ctypes.c_void_p
    fn.restype = ctypes.c_int
    fn.argtypes = [vp, vp, vp, vp, vp, vp, vp, ctypes.POINTER(rr.Dims), ctypes.c_float, vp, vp]
    return fn


def test_noalloc_matches_allocating_entry_point_on_two_calls():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as rr
    fn = _noalloc_fn(rr)
    # several agents, ragged Q tiles, a mid-page prefix and a prefix-less agent
    wl = synth.custom("noalloc", 4, 8, 2, 128, [300, 0, 1037, 64], [70, 150, 33, 257], seed=6)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    ref = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"])
    assert rr.device_error() == 0
    ref64 = to_f64(ref)
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
        d = np.abs(to_f64(out) - ref64)
        assert np.isfinite(d).all(), f"call {call}: non-finite output"
        assert d.max() <= MAX_ABS and d.mean() <= MEAN_ABS, f"call {call}: max {d.max():.3e} mean {d.mean():.3e}"


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

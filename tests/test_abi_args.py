"""Argument checks of the C ABI that run on the host before any device work (CPU only).

Every entry point validates its sizes, pointers and alignment first and returns an RR_ERR_* code
with a message, never aborting.  Here each call gets dims or pointers that fail one of those
checks; pointers are NULL or small integers that are never dereferenced, since the check fails
first.  A batch with no agents and no tokens returns RR_OK without touching a device.  The tests
skip on a machine with a GPU (the GPU suite covers the same errors with real buffers), so a check
that regressed can never send made-up pointers to a kernel.
"""
import ctypes
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

OK, INVALID, UNSUPPORTED = 0, 1, 2
A16, A4, MIS = 0x10000, 0x20000, 0x10008   # 16-byte aligned, 4-byte aligned, 8 but not 16-byte aligned


@pytest.fixture(scope="module")
def rr():
    import torch
    if torch.cuda.is_available():
        pytest.skip("host-side argument checks are tested on a machine without a GPU")
    import paper_2609_32278_gb300 as m
    if not os.path.exists(m._SO):
        pytest.skip("librr.so not built (run __graft_entry__.build())")
    m.lib()
    return m


def dims(rr, B=2, Hq=8, Hkv=2, D=128, ps=16, max_pages=4, num_pages=64, T=10):
    return ctypes.byref(rr.make_dims(B, Hq, Hkv, D, ps, max_pages, num_pages, T))


def attn(rr, d, q=A16, kp=A16, vp=A16, pt=A4, pl=A4, sl=A4, out=A16):
    return rr.lib().rr_extend_attention(q, kp, vp, pt, pl, sl, out, d, 0.0, None)


def append(rr, d, kn=A16, vn=A16, kp=A16, vp=A16, pt=A4, pl=A4, sl=A4):
    return rr.lib().rr_kv_append(kn, vn, kp, vp, pt, pl, sl, d, None)


def expect(rr, rc, code, words):
    assert rc == code, (rc, rr.last_error())
    msg = rr.last_error()
    for w in words:
        assert w in msg, msg


@pytest.mark.parametrize("kw,code,words", [
    (dict(B=-1), INVALID, ["negative"]),
    (dict(T=-5), INVALID, ["negative"]),
    (dict(Hq=6, Hkv=4), INVALID, ["multiple of num_kv_heads"]),
    (dict(Hkv=0), INVALID, ["num_kv_heads"]),
    (dict(D=96), UNSUPPORTED, ["head_dim 96"]),
    (dict(ps=12), UNSUPPORTED, ["page_size 12"]),
    (dict(ps=256), UNSUPPORTED, ["page_size 256"]),
    (dict(Hq=6, Hkv=2), UNSUPPORTED, ["GQA group 3"]),
    (dict(Hq=64, Hkv=2), UNSUPPORTED, ["GQA group 32"]),
    (dict(T=1 << 31), UNSUPPORTED, ["total_tokens"]),
    (dict(num_pages=1 << 27, ps=16), UNSUPPORTED, ["num_pages * page_size"]),
    (dict(max_pages=0), INVALID, ["max_pages is 0"]),
])
def test_attention_rejects_bad_dims(rr, kw, code, words):
    expect(rr, attn(rr, dims(rr, **kw)), code, words)


def test_append_takes_any_group_but_checks_the_rest(rr):
    # the append has no GQA packing: group 3 passes the size checks and fails on the NULL K pointer
    expect(rr, append(rr, dims(rr, Hq=6, Hkv=2), kn=None), INVALID, ["null K/V"])
    expect(rr, append(rr, dims(rr, D=96)), UNSUPPORTED, ["head_dim"])


def test_null_dims(rr):
    assert rr.lib().rr_extend_attention(A16, A16, A16, A4, A4, A4, A16, None, 0.0, None) == INVALID
    assert "dims is null" in rr.last_error()


@pytest.mark.parametrize("which", ["q", "kp", "vp", "out"])
def test_attention_null_buffer(rr, which):
    expect(rr, attn(rr, dims(rr), **{which: None}), INVALID, ["null q/pool/out"])


@pytest.mark.parametrize("which", ["pt", "pl", "sl"])
def test_attention_null_lengths(rr, which):
    expect(rr, attn(rr, dims(rr), **{which: None}), INVALID, ["null lens or page table"])


@pytest.mark.parametrize("which", ["q", "kp", "vp", "out"])
def test_attention_misaligned_buffer(rr, which):
    expect(rr, attn(rr, dims(rr), **{which: MIS}), INVALID, ["16-byte aligned"])


def test_attention_misaligned_lengths(rr):
    expect(rr, attn(rr, dims(rr), pl=A4 + 2), INVALID, ["4-byte aligned"])


def test_attention_empty_pool(rr):
    expect(rr, attn(rr, dims(rr, num_pages=0)), INVALID, ["empty pool"])


@pytest.mark.parametrize("which", ["kn", "vn", "kp", "vp"])
def test_append_null_and_misaligned(rr, which):
    expect(rr, append(rr, dims(rr), **{which: None}), INVALID, ["null K/V"])
    expect(rr, append(rr, dims(rr), **{which: MIS}), INVALID, ["16-byte aligned"])


def test_empty_batch_is_ok_everywhere(rr):
    L = rr.lib()
    d = dims(rr, B=0, T=0, max_pages=0, num_pages=0)
    assert attn(rr, d, None, None, None, None, None, None, None) == OK
    assert append(rr, d, None, None, None, None, None, None, None) == OK
    assert L.rr_extend_step(None, None, None, None, None, None, None, None, None, d, 0.0, None) == OK
    assert L.rr_decode_attention(None, None, None, None, None, None, d, 0.0, None) == OK
    assert L.rr_decode_attention_shared(None, None, None, None, None, 128, None, d, 0.0, None) == OK
    assert L.rr_rope_table(None, 0, 128, 500000.0, None) == OK


def test_decode_needs_one_token_per_agent(rr):
    L = rr.lib()
    rc = L.rr_decode_attention(A16, A16, A16, A4, A4, A16, dims(rr, B=3, T=4), 0.0, None)
    expect(rr, rc, INVALID, ["one query token per agent", "(4) != batch (3)"])
    rc = L.rr_decode_attention(A16, A16, A16, A4, None, A16, dims(rr, B=3, T=3), 0.0, None)
    expect(rr, rc, INVALID, ["null kv_lens"])


@pytest.mark.parametrize("shared_len,code,words", [
    (0, UNSUPPORTED, ["shared_len (0)"]),
    (100, UNSUPPORTED, ["multiple of 128"]),
    (128 * 8, INVALID, ["exceeds max_pages"]),   # 4 pages of 16 tokens hold 64 positions
])
def test_decode_shared_prefix_length(rr, shared_len, code, words):
    rc = rr.lib().rr_decode_attention_shared(A16, A16, A16, A4, A4, shared_len, A16, dims(rr, B=3, T=3), 0.0, None)
    expect(rr, rc, code, words)


def test_rope_entry_points_check_the_table(rr):
    L = rr.lib()
    d = dims(rr)
    expect(rr, L.rr_kv_append_rope(A16, A16, A16, A16, A4, A4, A4, d, None, 100, None), INVALID, ["null rope table"])
    expect(rr, L.rr_kv_append_rope(A16, A16, A16, A16, A4, A4, A4, d, MIS, 100, None), INVALID, ["rope table"])
    expect(rr, L.rr_kv_append_rope(A16, A16, A16, A16, A4, A4, A4, d, A16, 0, None), INVALID, ["rope_max_pos"])
    expect(rr, L.rr_extend_attention_rope(A16, A16, A16, A4, A4, A4, A16, d, 0.0, None, 100, None), INVALID,
           ["null rope table"])
    expect(rr, L.rr_decode_attention_rope(A16, A16, A16, A4, A4, A16, dims(rr, T=2), 0.0, None, 100, None), INVALID,
           ["null rope table"])
    expect(rr, L.rr_rope_table(A16, -1, 128, 500000.0, None), INVALID, ["max_pos"])
    expect(rr, L.rr_rope_table(A16, 10, 96, 500000.0, None), UNSUPPORTED, ["head_dim 96"])
    expect(rr, L.rr_rope_table(A16, 10, 128, 1.0, None), INVALID, ["base"])
    expect(rr, L.rr_rope_table(MIS, 10, 128, 500000.0, None), INVALID, ["16-byte aligned"])


def test_fused_step_needs_both_new_rows(rr):
    L = rr.lib()
    rc = L.rr_extend_step(A16, A16, None, A16, A16, A4, A4, A4, A16, dims(rr), 0.0, None)
    expect(rr, rc, INVALID, ["null k_new / v_new"])
    rc = L.rr_extend_step(A16, MIS, A16, A16, A16, A4, A4, A4, A16, dims(rr), 0.0, None)
    expect(rr, rc, INVALID, ["k_new / v_new must be 16-byte aligned"])


def test_error_message_is_cleared_by_a_good_call(rr):
    expect(rr, attn(rr, dims(rr, D=96)), UNSUPPORTED, ["head_dim"])
    assert attn(rr, dims(rr, B=0, T=0, max_pages=0, num_pages=0)) == OK
    assert rr.last_error() == ""


def shared_attn(rr, d, shared_len, q=A16, kp=A16, vp=A16, pt=A4, pl=A4, sl=A4, out=A16):
    return rr.lib().rr_extend_attention_shared(q, kp, vp, pt, pl, sl, shared_len, out, d, 0.0, None)


@pytest.mark.parametrize("shared_len,code,words", [
    (0, UNSUPPORTED, ["shared_len (0)", "multiple of 128"]),
    (-128, UNSUPPORTED, ["shared_len (-128)"]),
    (200, UNSUPPORTED, ["shared_len (200)"]),
    (128 * 5, INVALID, ["exceeds max_pages"]),       # 4 pages x 16 tokens
])
def test_shared_cascade_rejects_bad_shared_len(rr, shared_len, code, words):
    expect(rr, shared_attn(rr, dims(rr, max_pages=4), shared_len), code, words)


def test_shared_cascade_checks_like_the_plain_call(rr):
    expect(rr, shared_attn(rr, dims(rr, D=96), 128), UNSUPPORTED, ["head_dim 96"])
    expect(rr, shared_attn(rr, dims(rr, max_pages=8), 128, q=None), INVALID, ["null q/pool/out"])
    expect(rr, shared_attn(rr, dims(rr, max_pages=8), 128, pt=None), INVALID, ["null lens or page table"])
    expect(rr, shared_attn(rr, dims(rr, max_pages=8), 128, out=MIS), INVALID, ["16-byte aligned"])
    assert shared_attn(rr, dims(rr, B=0, T=0), 128) == OK

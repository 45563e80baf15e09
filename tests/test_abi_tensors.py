"""Host-side layout checks of the rr_tensor calls (rr_kv_append_tensors, rr_extend_attention_tensors), on a
machine without a GPU.

Each case describes the arguments of a small extend step (2 agents, 8 query / 2 KV heads, d128, 16-token
pages) with one argument wrong -- a strided or transposed view, a wrong element type, a wrong rank, shapes
that disagree -- and checks the code and the message; the data pointers are small aligned integers that
are never dereferenced, since every check runs before any device work.  Like the other host-side argument
tests, these skip on a machine with a GPU (tests/test_gpu_tensors.py runs the passing path there).
"""
import ctypes
import os

import pytest

OK, INVALID, UNSUPPORTED = 0, 1, 2
A16, A4 = 0x10000, 0x20000
BF16, I32 = 1, 2


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


def mk(rr, shape, dtype, data=A16, stride=None):
    t = rr.RRTensor()
    t.data = data
    t.ndim = len(shape)
    st, acc = [], 1
    for x in reversed(shape):
        st.append(acc)
        acc *= x
    st = list(reversed(st)) if stride is None else stride
    for i, (x, s) in enumerate(zip(shape, st)):
        t.shape[i] = x
        t.stride[i] = s
    t.dtype = dtype
    return t


def attn_args(rr, T=10, B=2):
    return dict(q=mk(rr, [T, 8, 128], BF16), k_pool=mk(rr, [64, 16, 2, 128], BF16),
                v_pool=mk(rr, [64, 16, 2, 128], BF16), page_table=mk(rr, [B, 4], I32, A4),
                prefix_lens=mk(rr, [B], I32, A4), suffix_lens=mk(rr, [B], I32, A4), out=mk(rr, [T, 8, 128], BF16))


def append_args(rr, T=10, B=2):
    return dict(k_new=mk(rr, [T, 2, 128], BF16), v_new=mk(rr, [T, 2, 128], BF16),
                k_pool=mk(rr, [64, 16, 2, 128], BF16), v_pool=mk(rr, [64, 16, 2, 128], BF16),
                page_table=mk(rr, [B, 4], I32, A4), prefix_lens=mk(rr, [B], I32, A4),
                suffix_lens=mk(rr, [B], I32, A4))


def call_attn(rr, a):
    ref = lambda k: None if a[k] is None else ctypes.byref(a[k])
    keys = ("q", "k_pool", "v_pool", "page_table", "prefix_lens", "suffix_lens", "out")
    return rr.lib().rr_extend_attention_tensors(*[ref(k) for k in keys], 0.0, None)


def call_append(rr, a):
    keys = ("k_new", "v_new", "k_pool", "v_pool", "page_table", "prefix_lens", "suffix_lens")
    return rr.lib().rr_kv_append_tensors(*[ctypes.byref(a[k]) for k in keys], None)


def expect(rr, rc, code, words):
    assert rc == code, (rc, rr.last_error())
    for w in words:
        assert w in rr.last_error(), rr.last_error()


ATTN_CASES = [
    # name, argument(s), replacement, code, words in the message
    ("q_strided_rows", "q", lambda rr: mk(rr, [10, 8, 128], BF16, stride=[2048, 128, 1]), UNSUPPORTED,
     ["q", "stride 2048", "dimension 0", "1024"]),
    ("q_heads_dims_transposed", "q", lambda rr: mk(rr, [10, 8, 128], BF16, stride=[1024, 1, 8]), UNSUPPORTED,
     ["q", "dimension 2"]),
    ("pool_slot_stride", "k_pool", lambda rr: mk(rr, [64, 16, 2, 128], BF16, stride=[8192, 512, 128, 1]),
     UNSUPPORTED, ["k_pool", "dimension 1"]),
    ("pool_int32", "v_pool", lambda rr: mk(rr, [64, 16, 2, 128], I32), UNSUPPORTED, ["v_pool", "dtype", "bf16"]),
    ("lens_bf16", "prefix_lens", lambda rr: mk(rr, [2], BF16, A4), UNSUPPORTED, ["prefix_lens", "int32"]),
    ("out_unknown_dtype", "out", lambda rr: mk(rr, [10, 8, 128], 7), UNSUPPORTED, ["out", "unknown"]),
    ("page_table_rank", "page_table", lambda rr: mk(rr, [8], I32, A4), INVALID, ["page_table", "1 dimensions"]),
    ("q_rank", "q", lambda rr: mk(rr, [10, 1024], BF16), INVALID, ["q", "expected 3"]),
    ("out_rows", "out", lambda rr: mk(rr, [11, 8, 128], BF16), INVALID, ["q dimension 0", "out"]),
    ("q_head_dim", ("q", "out"), lambda rr: mk(rr, [10, 8, 64], BF16), INVALID,
     ["q dimension 2", "k_pool dimension 3"]),
    ("v_pool_pages", "v_pool", lambda rr: mk(rr, [65, 16, 2, 128], BF16), INVALID, ["k_pool", "v_pool"]),
    ("suffix_lens_batch", "suffix_lens", lambda rr: mk(rr, [3], I32, A4), INVALID, ["suffix_lens", "page_table"]),
    ("negative_extent", "page_table", lambda rr: mk(rr, [2, -4], I32, A4), INVALID, ["negative"]),
    ("null_data", "q", lambda rr: mk(rr, [10, 8, 128], BF16, data=0), INVALID, ["q", "null data"]),
    ("null_tensor", "k_pool", lambda rr: None, INVALID, ["k_pool", "null rr_tensor"]),
]


@pytest.mark.parametrize("name,arg,repl,code,words", ATTN_CASES, ids=[c[0] for c in ATTN_CASES])
def test_attention_rejects(rr, name, arg, repl, code, words):
    a = attn_args(rr)
    for k in (arg if isinstance(arg, tuple) else (arg,)):
        a[k] = repl(rr)
    expect(rr, call_attn(rr, a), code, words)


APPEND_CASES = [
    ("k_new_strided", "k_new", lambda rr: mk(rr, [10, 2, 128], BF16, stride=[512, 128, 1]), UNSUPPORTED,
     ["k_new", "stride 512"]),
    ("v_new_int32", "v_new", lambda rr: mk(rr, [10, 2, 128], I32), UNSUPPORTED, ["v_new", "dtype"]),
    ("v_new_rows", "v_new", lambda rr: mk(rr, [9, 2, 128], BF16), INVALID, ["k_new", "v_new"]),
    ("k_new_heads", ("k_new", "v_new"), lambda rr: mk(rr, [10, 4, 128], BF16), INVALID,
     ["k_new dimension 1", "k_pool"]),
    ("pool_rank", "k_pool", lambda rr: mk(rr, [64, 16, 256], BF16), INVALID, ["k_pool", "expected 4"]),
]


@pytest.mark.parametrize("name,arg,repl,code,words", APPEND_CASES, ids=[c[0] for c in APPEND_CASES])
def test_append_rejects(rr, name, arg, repl, code, words):
    a = append_args(rr)
    for k in (arg if isinstance(arg, tuple) else (arg,)):
        a[k] = repl(rr)
    expect(rr, call_append(rr, a), code, words)


def test_empty_batch_is_ok_without_a_device(rr):
    a = attn_args(rr, T=0, B=0)
    assert call_attn(rr, a) == OK, rr.last_error()
    assert call_append(rr, append_args(rr, T=0, B=0)) == OK, rr.last_error()


def test_extent_one_dimensions_may_have_any_stride(rr):
    """A dimension of extent 1 is never stepped through, so its stride is not checked: the call passes every
    layout check and only then fails for want of a device."""
    a = attn_args(rr, T=1, B=1)
    a["q"] = mk(rr, [1, 8, 128], BF16, stride=[123456, 128, 1])
    a["prefix_lens"] = mk(rr, [1], I32, A4, stride=[7])
    rc = call_attn(rr, a)
    assert rc not in (INVALID, UNSUPPORTED), rr.last_error()

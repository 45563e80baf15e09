"""GB300 extend attention over a paged KV pool -- Python binding of librr.so.

Two calls make one extend step for a batch of returning agents (RR-Evict,
Sec. 1-2: reuse each agent's surviving cached prefix, prefill its uncached
suffix):

    kv_append(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens)
    out = extend_attention(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens)

With rotary position embedding (q and k_new un-rotated; rotated at positions P_b + j):

    rope = rope_table(max_pos, head_dim, base)
    out = extend_step(q, k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, rope=rope)

and the step after it, one new token per agent:

    kv_append(k_tok, v_tok, k_pool, v_pool, page_table, kv_lens - 1, ones)
    out = decode_attention(q_tok, k_pool, v_pool, page_table, kv_lens)

This module only marshals torch tensors into the C ABI of include/rr.h; every
step of the computation runs in the CUDA kernels of librr.so.  There is no
fallback: if the library is missing or a call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "librr.so")

RR_OK = 0
RR_ERR_INVALID_ARG = 1
RR_ERR_UNSUPPORTED = 2
RR_ERR_CUDA = 3
RR_ERR_TIMEOUT = 4
RR_ERR_OOB = 5
RR_ERR_LENS = 6
RR_ERR_OVERLAP = 7
RR_ERR_SHARED = 8

# Every symbol include/rr.h declares.
EXPORTS = ("rr_kv_append", "rr_extend_attention", "rr_extend_step", "rr_decode_attention", "rr_validate_page_table",
           "rr_get_device_error", "rr_last_error", "rr_version", "rr_shutdown", "rr_extend_attention_noalloc",
           "rr_rope_table", "rr_kv_append_rope", "rr_extend_attention_rope", "rr_extend_step_rope",
           "rr_decode_attention_rope", "rr_decode_attention_shared", "rr_set_wait_limit", "rr_kv_append_tensors",
           "rr_extend_attention_tensors", "rr_extend_attention_shared")

RR_DTYPE_BF16 = 1
RR_DTYPE_I32 = 2


class RRError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"rr error {code}: {msg}")
        self.code = code


class Dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32), ("max_pages", ctypes.c_int32),
                ("num_pages", ctypes.c_int64), ("total_tokens", ctypes.c_int64)]


class RRTensor(ctypes.Structure):
    """rr_tensor of include/rr.h: data pointer, rank, shape and strides (in elements), element type."""
    _fields_ = [("data", ctypes.c_void_p), ("ndim", ctypes.c_int32), ("shape", ctypes.c_int64 * 4),
                ("stride", ctypes.c_int64 * 4), ("dtype", ctypes.c_int32)]


_lib = None


def build(verbose: bool = False) -> str:
    from . import native_build
    return native_build.build(verbose=verbose)


def lib():
    """The loaded librr.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_SO):
            raise RuntimeError(f"{_SO} not found: build it with __graft_entry__.build() "
                               "(there is no fallback implementation)")
        L = ctypes.CDLL(_SO)
        vp = ctypes.c_void_p
        dp = ctypes.POINTER(Dims)
        L.rr_kv_append.restype = ctypes.c_int
        L.rr_kv_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, dp, vp]
        L.rr_extend_attention.restype = ctypes.c_int
        L.rr_extend_attention.argtypes = [vp, vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp]
        L.rr_extend_step.restype = ctypes.c_int
        L.rr_extend_step.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp]
        L.rr_decode_attention.restype = ctypes.c_int
        L.rr_decode_attention.argtypes = [vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp]
        L.rr_rope_table.restype = ctypes.c_int
        L.rr_rope_table.argtypes = [vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_double, vp]
        L.rr_kv_append_rope.restype = ctypes.c_int
        L.rr_kv_append_rope.argtypes = [vp, vp, vp, vp, vp, vp, vp, dp, vp, ctypes.c_int32, vp]
        L.rr_extend_attention_rope.restype = ctypes.c_int
        L.rr_extend_attention_rope.argtypes = [vp, vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp, ctypes.c_int32, vp]
        L.rr_extend_step_rope.restype = ctypes.c_int
        L.rr_extend_step_rope.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp, ctypes.c_int32,
                                          vp]
        L.rr_extend_attention_shared.restype = ctypes.c_int
        L.rr_extend_attention_shared.argtypes = [vp, vp, vp, vp, vp, vp, ctypes.c_int32, vp, dp, ctypes.c_float, vp]
        L.rr_decode_attention_shared.restype = ctypes.c_int
        L.rr_decode_attention_shared.argtypes = [vp, vp, vp, vp, vp, ctypes.c_int32, vp, dp, ctypes.c_float, vp]
        L.rr_decode_attention_rope.restype = ctypes.c_int
        L.rr_decode_attention_rope.argtypes = [vp, vp, vp, vp, vp, vp, dp, ctypes.c_float, vp, ctypes.c_int32, vp]
        L.rr_validate_page_table.restype = ctypes.c_int
        L.rr_validate_page_table.argtypes = [vp, vp, vp, dp]
        L.rr_get_device_error.restype = ctypes.c_int
        L.rr_get_device_error.argtypes = [vp]
        L.rr_last_error.restype = ctypes.c_char_p
        L.rr_last_error.argtypes = []
        L.rr_version.restype = ctypes.c_char_p
        L.rr_version.argtypes = []
        L.rr_set_wait_limit.restype = None
        L.rr_set_wait_limit.argtypes = [ctypes.c_longlong]
        tp = ctypes.POINTER(RRTensor)
        L.rr_kv_append_tensors.restype = ctypes.c_int
        L.rr_kv_append_tensors.argtypes = [tp] * 7 + [vp]
        L.rr_extend_attention_tensors.restype = ctypes.c_int
        L.rr_extend_attention_tensors.argtypes = [tp] * 7 + [ctypes.c_float, vp]
        L.rr_shutdown.restype = None
        L.rr_shutdown.argtypes = []
        _lib = L
    return _lib


def _check(rc: int) -> None:
    if rc != RR_OK:
        raise RRError(rc, lib().rr_last_error().decode(errors="replace"))


def _stream_ptr(stream, device):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, name, dtype, ndim):
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def make_dims(B, Hq, Hkv, D, ps, max_pages, num_pages, T) -> Dims:
    return Dims(int(B), int(Hq), int(Hkv), int(D), int(ps), int(max_pages), int(num_pages), int(T))


def rope_table(max_pos: int, head_dim: int, base: float, device=None, stream=None):
    """(cos, sin) table of the rotary embedding, float32 [max_pos, head_dim // 2, 2] (rr_rope_table)."""
    import torch
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    table = torch.empty((int(max_pos), int(head_dim) // 2, 2), dtype=torch.float32, device=dev)
    _check(lib().rr_rope_table(table.data_ptr(), int(max_pos), int(head_dim), float(base), _stream_ptr(stream, dev)))
    return table


def _rope_arg(rope, D):
    """(pointer, max_pos) of a rope_table() tensor, or None."""
    import torch
    if rope is None:
        return None
    _need(rope, "rope", torch.float32, 3)
    if rope.shape[1:] != (D // 2, 2):
        raise ValueError(f"rope table must be [max_pos, {D // 2}, 2] for head dim {D}, got {tuple(rope.shape)}")
    return rope.data_ptr(), int(rope.shape[0])


def kv_append(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, stream=None, rope=None) -> None:
    """Write suffix K/V rows into their pool slots (rr_kv_append); with a rope table, K is rotated at its
    positions on the way (rr_kv_append_rope)."""
    import torch
    _need(k_new, "k_new", torch.bfloat16, 3)
    _need(v_new, "v_new", torch.bfloat16, 3)
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(page_table, "page_table", torch.int32, 2)
    _need(prefix_lens, "prefix_lens", torch.int32, 1)
    _need(suffix_lens, "suffix_lens", torch.int32, 1)
    T, Hkv, D = k_new.shape
    num_pages, ps, Hkv2, D2 = k_pool.shape
    if v_new.shape != k_new.shape or v_pool.shape != k_pool.shape or (Hkv2, D2) != (Hkv, D):
        raise ValueError("k/v shapes disagree")
    B = prefix_lens.shape[0]
    if suffix_lens.shape[0] != B or page_table.shape[0] != B:
        raise ValueError("lens / page_table batch sizes disagree")
    dims = make_dims(B, Hkv, Hkv, D, ps, page_table.shape[1], num_pages, T)
    args = (k_new.data_ptr(), v_new.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(), page_table.data_ptr(),
            prefix_lens.data_ptr(), suffix_lens.data_ptr(), ctypes.byref(dims))
    r = _rope_arg(rope, D)
    if r is None:
        _check(lib().rr_kv_append(*args, _stream_ptr(stream, k_new.device)))
    else:
        _check(lib().rr_kv_append_rope(*args, r[0], r[1], _stream_ptr(stream, k_new.device)))


def extend_attention(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, out=None,
                     softmax_scale: float = 0.0, stream=None, rope=None, shared_len: int = 0):
    """Extend attention of every suffix row over its agent's prefix + suffix (rr_extend_attention); with a
    rope table, each q row is rotated at its position first (rr_extend_attention_rope); with shared_len > 0,
    every agent's first shared_len positions are the same pages and the call runs as a cascade over them
    (rr_extend_attention_shared)."""
    import torch
    _need(q, "q", torch.bfloat16, 3)
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(page_table, "page_table", torch.int32, 2)
    _need(prefix_lens, "prefix_lens", torch.int32, 1)
    _need(suffix_lens, "suffix_lens", torch.int32, 1)
    T, Hq, D = q.shape
    num_pages, ps, Hkv, D2 = k_pool.shape
    if v_pool.shape != k_pool.shape or D2 != D:
        raise ValueError("q / pool shapes disagree")
    B = prefix_lens.shape[0]
    if suffix_lens.shape[0] != B or page_table.shape[0] != B:
        raise ValueError("lens / page_table batch sizes disagree")
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", torch.bfloat16, 3)
        if out.shape != q.shape:
            raise ValueError("out must have q's shape")
    dims = make_dims(B, Hq, Hkv, D, ps, page_table.shape[1], num_pages, T)
    args = (q.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(), page_table.data_ptr(), prefix_lens.data_ptr(),
            suffix_lens.data_ptr(), out.data_ptr(), ctypes.byref(dims), float(softmax_scale))
    r = _rope_arg(rope, D)
    if shared_len:
        if r is not None:
            raise ValueError("the shared-prefix cascade takes rotated queries only")
        _check(lib().rr_extend_attention_shared(q.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(),
                                                page_table.data_ptr(), prefix_lens.data_ptr(), suffix_lens.data_ptr(),
                                                int(shared_len), out.data_ptr(), ctypes.byref(dims),
                                                float(softmax_scale), _stream_ptr(stream, q.device)))
    elif r is None:
        _check(lib().rr_extend_attention(*args, _stream_ptr(stream, q.device)))
    else:
        _check(lib().rr_extend_attention_rope(*args, r[0], r[1], _stream_ptr(stream, q.device)))
    return out


def extend_step(q, k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, out=None,
                softmax_scale: float = 0.0, stream=None, rope=None):
    """kv_append + extend_attention in one attention launch (rr_extend_step): same pools, same output.
    With a rope table: the rotated append and the rotated attention (rr_extend_step_rope)."""
    import torch
    _need(q, "q", torch.bfloat16, 3)
    _need(k_new, "k_new", torch.bfloat16, 3)
    _need(v_new, "v_new", torch.bfloat16, 3)
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(page_table, "page_table", torch.int32, 2)
    _need(prefix_lens, "prefix_lens", torch.int32, 1)
    _need(suffix_lens, "suffix_lens", torch.int32, 1)
    T, Hq, D = q.shape
    num_pages, ps, Hkv, D2 = k_pool.shape
    if v_pool.shape != k_pool.shape or D2 != D or k_new.shape != (T, Hkv, D) or v_new.shape != k_new.shape:
        raise ValueError("q / k_new / v_new / pool shapes disagree")
    B = prefix_lens.shape[0]
    if suffix_lens.shape[0] != B or page_table.shape[0] != B:
        raise ValueError("lens / page_table batch sizes disagree")
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", torch.bfloat16, 3)
        if out.shape != q.shape:
            raise ValueError("out must have q's shape")
    dims = make_dims(B, Hq, Hkv, D, ps, page_table.shape[1], num_pages, T)
    args = (q.data_ptr(), k_new.data_ptr(), v_new.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(),
            page_table.data_ptr(), prefix_lens.data_ptr(), suffix_lens.data_ptr(), out.data_ptr(), ctypes.byref(dims),
            float(softmax_scale))
    r = _rope_arg(rope, D)
    if r is None:
        _check(lib().rr_extend_step(*args, _stream_ptr(stream, q.device)))
    else:
        _check(lib().rr_extend_step_rope(*args, r[0], r[1], _stream_ptr(stream, q.device)))
    return out


def decode_attention(q, k_pool, v_pool, page_table, kv_lens, out=None, softmax_scale: float = 0.0, stream=None,
                     rope=None, shared_len: int = 0):
    """Decode attention: the one new query token of each agent over its kv_lens[b] keys (rr_decode_attention).

    q: [B, Hq, D] bf16; kv_lens: [B] int32, the new token's K/V already appended.  With a rope table, q is
    rotated at position kv_lens[b] - 1 first (rr_decode_attention_rope).  shared_len > 0: every agent's first
    shared_len positions are the same pages, read once per group of agents (rr_decode_attention_shared)."""
    import torch
    _need(q, "q", torch.bfloat16, 3)
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(page_table, "page_table", torch.int32, 2)
    _need(kv_lens, "kv_lens", torch.int32, 1)
    B, Hq, D = q.shape
    num_pages, ps, Hkv, D2 = k_pool.shape
    if v_pool.shape != k_pool.shape or D2 != D:
        raise ValueError("q / pool shapes disagree")
    if kv_lens.shape[0] != B or page_table.shape[0] != B:
        raise ValueError("q / kv_lens / page_table batch sizes disagree")
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", torch.bfloat16, 3)
        if out.shape != q.shape:
            raise ValueError("out must have q's shape")
    dims = make_dims(B, Hq, Hkv, D, ps, page_table.shape[1], num_pages, B)
    args = (q.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(), page_table.data_ptr(), kv_lens.data_ptr(),
            out.data_ptr(), ctypes.byref(dims), float(softmax_scale))
    r = _rope_arg(rope, D)
    if shared_len:
        if r is not None:
            raise ValueError("the shared-prefix decode takes rotated queries only")
        _check(lib().rr_decode_attention_shared(q.data_ptr(), k_pool.data_ptr(), v_pool.data_ptr(),
                                                page_table.data_ptr(), kv_lens.data_ptr(), int(shared_len),
                                                out.data_ptr(), ctypes.byref(dims), float(softmax_scale),
                                                _stream_ptr(stream, q.device)))
    elif r is None:
        _check(lib().rr_decode_attention(*args, _stream_ptr(stream, q.device)))
    else:
        _check(lib().rr_decode_attention_rope(*args, r[0], r[1], _stream_ptr(stream, q.device)))
    return out


def tensor_arg(t) -> RRTensor:
    """The rr_tensor of a torch tensor as it is (its real strides and element type, not a checked copy), so
    that the library's own layout checks see what the caller passes."""
    import torch
    codes = {torch.bfloat16: RR_DTYPE_BF16, torch.int32: RR_DTYPE_I32}
    if t.dim() > 4:
        raise ValueError(f"rr_tensor holds at most 4 dimensions, got {t.dim()}")
    r = RRTensor()
    r.data = t.data_ptr()
    r.ndim = t.dim()
    for i in range(t.dim()):
        r.shape[i] = int(t.shape[i])
        r.stride[i] = int(t.stride(i))
    r.dtype = codes.get(t.dtype, 0)
    return r


def kv_append_tensors(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, stream=None) -> None:
    """rr_kv_append_tensors: the append with every argument's shape, strides and type checked by the library."""
    ts = [tensor_arg(t) for t in (k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens)]
    _check(lib().rr_kv_append_tensors(*[ctypes.byref(t) for t in ts], _stream_ptr(stream, k_new.device)))


def extend_attention_tensors(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, out,
                             softmax_scale: float = 0.0, stream=None):
    """rr_extend_attention_tensors: the attention with every argument's shape, strides and type checked by
    the library."""
    ts = [tensor_arg(t) for t in (q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, out)]
    _check(lib().rr_extend_attention_tensors(*[ctypes.byref(t) for t in ts], float(softmax_scale),
                                             _stream_ptr(stream, q.device)))
    return out


def device_error(stream=None, device=None) -> int:
    """Synchronise the stream and return (and clear) the device error word."""
    import torch
    dev = device if device is not None else torch.device("cuda", torch.cuda.current_device())
    return int(lib().rr_get_device_error(_stream_ptr(stream, dev)))


def validate_page_table(page_table, prefix_lens, suffix_lens, num_pages: int, page_size: int,
                        total_tokens: Optional[int] = None) -> int:
    """Host-side page-table check (numpy int32 arrays); returns an RR_* code, never raises on bad tables."""
    import numpy as np
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    pl = np.ascontiguousarray(prefix_lens, dtype=np.int32)
    sl = np.ascontiguousarray(suffix_lens, dtype=np.int32)
    T = int(sl.sum()) if total_tokens is None else int(total_tokens)
    dims = make_dims(len(pl), 1, 1, 64, page_size, pt.shape[1] if pt.ndim == 2 else 0, num_pages, T)
    return int(lib().rr_validate_page_table(pt.ctypes.data, pl.ctypes.data, sl.ctypes.data, ctypes.byref(dims)))


def set_wait_limit(cycles: int) -> None:
    """Budget in clock cycles of the decode kernel's pipeline waits and the extend kernel's stage-watcher
    waits (<= 0: the default, ~4 s); a wait that runs out ends the kernel with RR_ERR_TIMEOUT in the
    device error word (rr_set_wait_limit)."""
    lib().rr_set_wait_limit(int(cycles))


def last_error() -> str:
    return lib().rr_last_error().decode(errors="replace")


def version() -> str:
    return lib().rr_version().decode()

"""fp64 CPU oracle for the extend-attention path -- TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package.  It shares no code with the CUDA library and never
takes an input or an expected value from it.  The arithmetic lives in
rr_oracle.c (plain loops, double precision); this file only builds it and
marshals numpy arrays.

Readings of the paper used here (it never writes the attention formula):
* append: suffix token j of agent b lands at position P_b + j, page
  page_table[b][pos // ps], slot pos % ps (Sec. 2, "materializes their KV
  tensors" into the shared pool);
* attention: causal, aligned bottom-right -- suffix row i of agent b sees all
  P_b cached keys and the suffix keys up to and including itself (Sec. 1,
  Sec. 2: reuse the cached prefix, compute the uncached suffix);
* GQA: query head h reads KV head h // (Hq // Hkv);
* rotary position embedding (not in the paper; the models its agents run use it): the suffix's q and
  k rows are rotated at their absolute positions P_b + j, rotate-half pairing (dim i with i + D/2),
  angle p * base^(-2i/D); q is used unrounded, a rotated K row is rounded once to the pool's bf16.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "librr_oracle.so")

OK, BAD_ARG, BAD_PAGE, NO_MEM = 0, 1, 2, 3


def build(verbose: bool = False) -> None:
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-std=c11",
           os.path.join(_HERE, "rr_oracle.c"), "-o", _SO, "-lm"]
    if verbose:
        print(" ".join(cmd))
    subprocess.run(cmd, check=True)


_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(_SO):
            build()
        L = ctypes.CDLL(_SO)
        vp, i32, i64, f64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        L.oracle_kv_append.restype = ctypes.c_int
        L.oracle_kv_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i64]
        L.oracle_extend_attention.restype = ctypes.c_int
        L.oracle_extend_attention.argtypes = [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i64, f64,
                                              vp, vp, vp, i32]
        L.oracle_attention_rows.restype = ctypes.c_int
        L.oracle_attention_rows.argtypes = [vp, vp, i64, vp, vp, i64, i32, i32, f64, vp, vp, vp, i32]
        L.oracle_extend_attention_q64.restype = ctypes.c_int
        L.oracle_extend_attention_q64.argtypes = L.oracle_extend_attention.argtypes
        L.oracle_attention_rows_q64.restype = ctypes.c_int
        L.oracle_attention_rows_q64.argtypes = L.oracle_attention_rows.argtypes
        L.oracle_rope.restype = ctypes.c_int
        L.oracle_rope.argtypes = [vp, vp, i64, i32, i32, f64, vp]
        L.oracle_round_bf16.restype = ctypes.c_int
        L.oracle_round_bf16.argtypes = [vp, i64, vp]
        _lib = L
    return _lib


class OracleError(RuntimeError):
    pass


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _p(a):
    return a.ctypes.data if a is not None else None


def _threads(n):
    return n if n and n > 0 else (os.cpu_count() or 1)


def kv_append(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens):
    """Returns new (k_pool, v_pool) uint16 arrays with the suffix rows written (inputs are not modified)."""
    k_new, v_new = _c(k_new, np.uint16), _c(v_new, np.uint16)
    kp, vp = np.array(k_pool, dtype=np.uint16, copy=True), np.array(v_pool, dtype=np.uint16, copy=True)
    pt, pl, sl = _c(page_table, np.int32), _c(prefix_lens, np.int32), _c(suffix_lens, np.int32)
    num_pages, ps, Hkv, D = kp.shape
    rc = lib().oracle_kv_append(_p(k_new), _p(v_new), _p(kp), _p(vp), _p(pt), _p(pl), _p(sl), len(pl), Hkv, D,
                                ps, pt.shape[1], num_pages)
    if rc:
        raise OracleError(f"oracle_kv_append: {rc}")
    return kp, vp


def extend_attention(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, scale=None, nthreads=0,
                     with_stats=False):
    """out [T, Hq, D] float64 (and lse, wsum [T, Hq] if with_stats) from bf16-bit inputs.

    q may also be a float64 array (a q rotated by ``rope``, not rounded): it is then used as is."""
    q64 = np.asarray(q).dtype == np.float64
    q = _c(q, np.float64 if q64 else np.uint16)
    kp, vp = _c(k_pool, np.uint16), _c(v_pool, np.uint16)
    pt, pl, sl = _c(page_table, np.int32), _c(prefix_lens, np.int32), _c(suffix_lens, np.int32)
    T, Hq, D = q.shape
    num_pages, ps, Hkv, D2 = kp.shape
    assert D2 == D and int(sl.sum()) == T
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    out = np.zeros((T, Hq, D), dtype=np.float64)
    lse = np.zeros((T, Hq), dtype=np.float64) if with_stats else None
    wsum = np.zeros((T, Hq), dtype=np.float64) if with_stats else None
    fn = lib().oracle_extend_attention_q64 if q64 else lib().oracle_extend_attention
    rc = fn(_p(q), _p(kp), _p(vp), _p(pt), _p(pl), _p(sl), len(pl), Hq, Hkv, D, ps, pt.shape[1], num_pages,
            float(scale), _p(out), _p(lse), _p(wsum), _threads(nthreads))
    if rc:
        raise OracleError(f"oracle_extend_attention: {rc}")
    return (out, lse, wsum) if with_stats else out


def decode_attention(q, k_pool, v_pool, page_table, kv_lens, scale=None, nthreads=0, with_stats=False):
    """Decode attention: out [B, Hq, D] float64 -- the extend definition (Sec. 2) for a suffix of one token
    per agent.  Row b is agent b's new token, at position kv_lens[b] - 1; it sees all kv_lens[b] keys.

    No arithmetic of its own: the lengths are restated (prefix = L - 1, suffix = 1) and the extend
    oracle computes the plain definition."""
    L = _c(kv_lens, np.int32)
    if (L < 1).any():
        raise OracleError("decode_attention: every agent needs at least its own key")
    return extend_attention(q, k_pool, v_pool, page_table, L - 1, np.ones_like(L), scale=scale, nthreads=nthreads,
                            with_stats=with_stats)


def attention_rows(q_rows, positions, K, V, scale, nthreads=0, with_stats=False):
    """Selected rows of one agent / one KV group over its logical K, V ([n_keys, D] bf16 bits).

    q_rows: [n, G, D] bf16 bits (or float64, used as is); positions: [n] absolute positions.
    Returns out [n, G, D] float64.
    """
    q64 = np.asarray(q_rows).dtype == np.float64
    q_rows = _c(q_rows, np.float64 if q64 else np.uint16)
    positions = _c(positions, np.int64)
    K, V = _c(K, np.uint16), _c(V, np.uint16)
    n, G, D = q_rows.shape
    out = np.zeros((n, G, D), dtype=np.float64)
    lse = np.zeros((n, G), dtype=np.float64) if with_stats else None
    wsum = np.zeros((n, G), dtype=np.float64) if with_stats else None
    fn = lib().oracle_attention_rows_q64 if q64 else lib().oracle_attention_rows
    rc = fn(_p(q_rows), _p(positions), n, _p(K), _p(V), K.shape[0], G, D, float(scale), _p(out), _p(lse), _p(wsum),
            _threads(nthreads))
    if rc:
        raise OracleError(f"oracle_attention_rows: {rc}")
    return (out, lse, wsum) if with_stats else out


# ------------------------------------------------------------------ rotary position embedding (C)

def widen_bf16(bits):
    """bf16 bit patterns -> float64, exactly (the bits are the top half of a binary32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(x):
    """Nearest bf16 (ties to even) of float64 values, in one rounding; returns uint16 bit patterns."""
    x = _c(x, np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    rc = lib().oracle_round_bf16(_p(x), x.size, _p(out))
    if rc:
        raise OracleError(f"oracle_round_bf16: {rc}")
    return out


def rope(x, positions, base):
    """Rotate rows [n, heads, D] (bf16 bits or float64) at absolute positions [n]: float64 [n, heads, D].

    Rotate-half pairing (dim i with i + D/2), angle p * base^(-2i/D) for pair i (RoFormer's rotation,
    GPT-NeoX / Llama's pairing); see section (C) of rr_oracle.c."""
    x = np.asarray(x)
    x = _c(x, np.float64) if x.dtype == np.float64 else widen_bf16(x)
    pos = _c(positions, np.int64)
    n, heads, D = x.shape
    assert pos.shape == (n,)
    out = np.empty_like(x)
    rc = lib().oracle_rope(_p(x), _p(pos), n, heads, D, float(base), _p(out))
    if rc:
        raise OracleError(f"oracle_rope: {rc}")
    return out


def suffix_positions(prefix_lens, suffix_lens):
    """Absolute position of every packed suffix row: P_b + j for agent b's row j, agents in order."""
    pl = np.asarray(prefix_lens, dtype=np.int64)
    sl = np.asarray(suffix_lens, dtype=np.int64)
    return np.concatenate([p + np.arange(s, dtype=np.int64) for p, s in zip(pl, sl)] or [np.zeros(0, np.int64)])


def kv_append_rope(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, base):
    """kv_append of the suffix's K rotated at its positions (rounded once to the pool's bf16), V as is."""
    k_rot = round_bf16(rope(k_new, suffix_positions(prefix_lens, suffix_lens), base))
    return kv_append(k_rot, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens)


def extend_attention_rope(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, base, scale=None, nthreads=0,
                          with_stats=False):
    """extend_attention with q rotated at its positions in double precision (not rounded); the pool holds
    the rotated keys (kv_append_rope)."""
    q64 = rope(q, suffix_positions(prefix_lens, suffix_lens), base)
    return extend_attention(q64, k_pool, v_pool, page_table, prefix_lens, suffix_lens, scale=scale,
                            nthreads=nthreads, with_stats=with_stats)


def decode_attention_rope(q, k_pool, v_pool, page_table, kv_lens, base, scale=None, nthreads=0, with_stats=False):
    """decode_attention with each agent's query rotated at its position kv_lens[b] - 1 (no arithmetic of its
    own: the lengths are restated and extend_attention_rope computes it)."""
    L = _c(kv_lens, np.int32)
    if (L < 1).any():
        raise OracleError("decode_attention_rope: every agent needs at least its own key")
    return extend_attention_rope(q, k_pool, v_pool, page_table, L - 1, np.ones_like(L), base, scale=scale,
                                 nthreads=nthreads, with_stats=with_stats)


"""Seeded synthetic inputs for the extend-attention path.

This package holds no arithmetic of the attention or append method.  It makes
the inputs that the oracle harness and the GPU path both consume:

* per-agent cached-prefix / uncached-suffix lengths for the five workload
  shapes (agent-shaped batches standing in for the tau^2-bench and SWE-bench
  traces of Sec. 4, which are not available here);
* the page placement (a seeded Fisher-Yates permutation of the pool);
* the bf16 values of q, k_new, v_new and the cached prefix in the pool, each a
  pure function of its logical coordinates (see synth.c for the definition),
  generated either on the CPU (libsynth.so) or straight into device memory
  (libsynth_cuda.so, same definition, bit-identical).

Nothing here imports the product package or the oracle.
"""
from __future__ import annotations

import ctypes
import dataclasses
import hashlib
import json
import os
import subprocess
from typing import Dict, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_CPU_SO = os.path.join(_HERE, "libsynth.so")
_CUDA_SO = os.path.join(_HERE, "libsynth_cuda.so")

TENSOR_Q, TENSOR_K, TENSOR_V = 1, 2, 3
BF16_NAN = 0x7FC0          # quiet NaN: fills every pool slot no agent owns
MIX_GOLDEN = 0x9E3779B97F4A7C15
_U64 = (1 << 64) - 1


# --------------------------------------------------------------------------- build

def build(cuda: bool = True, verbose: bool = False) -> None:
    """Compile libsynth.so (gcc) and, if `cuda`, libsynth_cuda.so (nvcc, sm_103a)."""
    cmds = [["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-std=c11",
             os.path.join(_HERE, "synth.c"), "-o", _CPU_SO]]
    if cuda:
        cmds.append(["nvcc", "-O3", "-shared", "-Xcompiler", "-fPIC", "-std=c++17",
                     "-gencode", "arch=compute_103a,code=sm_103a", "-lineinfo",
                     os.path.join(_HERE, "synth_fill.cu"), "-o", _CUDA_SO])
    for c in cmds:
        if verbose:
            print(" ".join(c))
        subprocess.run(c, check=True)


_cpu_lib = None
_cuda_lib = None


def cpu_lib():
    global _cpu_lib
    if _cpu_lib is None:
        if not os.path.exists(_CPU_SO):
            build(cuda=False)
        lib = ctypes.CDLL(_CPU_SO)
        u64, i64, i32, u32 = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint32
        vp = ctypes.c_void_p
        lib.rrs_mix64.restype = u64
        lib.rrs_mix64.argtypes = [u64]
        lib.rrs_value.restype = ctypes.c_uint16
        lib.rrs_value.argtypes = [u64, u32, u32, u64, u32, u32]
        lib.rrs_fill_rows.restype = None
        lib.rrs_fill_rows.argtypes = [vp, vp, vp, i64, i32, i32, i32, u32, u64, i64, i32]
        lib.rrs_fill_pool_prefix.restype = None
        lib.rrs_fill_pool_prefix.argtypes = [vp, vp, vp, vp, i32, i32, i32, i32, i32, u64, i64, i32]
        lib.rrs_permutation.restype = None
        lib.rrs_permutation.argtypes = [vp, i64, u64]
        lib.rrs_stream.restype = None
        lib.rrs_stream.argtypes = [vp, i64, u64]
        _cpu_lib = lib
    return _cpu_lib


def cuda_lib():
    global _cuda_lib
    if _cuda_lib is None:
        if not os.path.exists(_CUDA_SO):
            raise RuntimeError(f"{_CUDA_SO} is missing: run synth.build() (or __graft_entry__.build())")
        lib = ctypes.CDLL(_CUDA_SO)
        vp, i64, i32, u32, u64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint32, ctypes.c_uint64
        lib.rrs_cuda_fill_rows.restype = ctypes.c_int
        lib.rrs_cuda_fill_rows.argtypes = [vp, vp, vp, i64, i32, i32, i32, u32, u64, i64, vp]
        lib.rrs_cuda_fill_pool.restype = ctypes.c_int
        lib.rrs_cuda_fill_pool.argtypes = [vp, vp, vp, vp, vp, i64, i32, i32, i32, u32, u64, i64, vp]
        _cuda_lib = lib
    return _cuda_lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


# --------------------------------------------------------------------------- seeded draws

def stream(n: int, seed: int) -> np.ndarray:
    """n SplitMix64 outputs starting from state `seed`."""
    out = np.empty(n, dtype=np.uint64)
    if n:
        cpu_lib().rrs_stream(_ptr(out), n, seed & _U64)
    return out


def uniform_ints(n: int, lo: int, hi: int, seed: int) -> np.ndarray:
    """n integers uniform in [lo, hi] (multiply-high reduction of SplitMix64 words)."""
    words = stream(n, seed)
    span = hi - lo + 1
    return np.array([lo + ((int(w) * span) >> 64) for w in words], dtype=np.int64)


def permutation(n: int, seed: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    if n:
        cpu_lib().rrs_permutation(_ptr(out), n, seed & _U64)
    return out


# --------------------------------------------------------------------------- workloads

@dataclasses.dataclass
class Workload:
    """Shapes, lengths and page placement of one extend batch.

    Layouts (all row-major): q/out [T, Hq, D] bf16; k_new/v_new [T, Hkv, D] bf16;
    k_pool/v_pool [num_pages, ps, Hkv, D] bf16; page_table [B, max_pages] int32
    (-1 past an agent's last page); prefix_lens/suffix_lens [B] int32.
    Agent b's suffix rows are q[cu[b]:cu[b+1]], cu = exclusive cumsum of suffix_lens.
    """
    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    ps: int
    prefix_lens: np.ndarray
    suffix_lens: np.ndarray
    shared_len: int
    num_pages: int
    page_table: np.ndarray
    seed: int

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def T(self) -> int:
        return int(self.suffix_lens.sum())

    @property
    def max_pages(self) -> int:
        return int(self.page_table.shape[1])

    @property
    def cu(self) -> np.ndarray:
        cu = np.zeros(self.B + 1, dtype=np.int64)
        np.cumsum(self.suffix_lens.astype(np.int64), out=cu[1:])
        return cu

    def manifest(self) -> Dict[str, object]:
        """What makes this batch reproducible: its name, seed and shapes, the per-agent lengths and a
        SHA-256 over the seed, every shape field, the lengths and the page table (the tensor values are a
        pure function of the seed and the logical coordinates, so these fix every input byte)."""
        fields = {"seed": int(self.seed), "B": int(self.B), "Hq": int(self.Hq), "Hkv": int(self.Hkv),
                  "D": int(self.D), "page_size": int(self.ps), "num_pages": int(self.num_pages),
                  "max_pages": self.max_pages, "shared_len": int(self.shared_len), "T": self.T}
        h = hashlib.sha256()
        h.update(json.dumps(fields, sort_keys=True).encode())
        for a in (self.prefix_lens, self.suffix_lens, self.page_table):
            arr = np.ascontiguousarray(a, dtype=np.int32)
            h.update(str(arr.shape).encode())
            h.update(arr.tobytes())
        return {"name": self.name, **fields,
                "prefix_lens": [int(x) for x in self.prefix_lens], "suffix_lens": [int(x) for x in self.suffix_lens],
                "sha256": h.hexdigest()}

    def write_manifest(self, path: str) -> str:
        """Write manifest() as JSON; returns its sha256."""
        m = self.manifest()
        with open(path, "w") as f:
            json.dump(m, f, indent=1)
            f.write("\n")
        return str(m["sha256"])

    def row_agent_pos(self):
        """(agent, absolute position) of every suffix row, in q's row order."""
        agent = np.repeat(np.arange(self.B, dtype=np.int32), self.suffix_lens.astype(np.int64))
        pos = np.concatenate([np.arange(int(p), int(p) + int(s), dtype=np.int64)
                              for p, s in zip(self.prefix_lens, self.suffix_lens)]) if self.T else \
            np.zeros(0, dtype=np.int64)
        return agent, pos


def place_pages(prefix_lens, suffix_lens, ps: int, num_pages: int, shared_len: int, seed: int,
                extra_cols: int = 0) -> np.ndarray:
    """Page table from a seeded permutation of the pool.

    Positions below `shared_len` (a whole number of pages) map to one common set
    of physical pages for every agent; every other page of every agent is a
    distinct physical page, taken from the permutation in agent order, then
    logical order.  Columns past an agent's last page hold -1.
    """
    assert shared_len % ps == 0
    B = len(prefix_lens)
    need = [-(-(int(p) + int(s)) // ps) for p, s in zip(prefix_lens, suffix_lens)]
    n_shared = shared_len // ps
    max_pages = max([1] + need) + extra_cols
    private = sum(max(0, n - n_shared) for n in need)
    if n_shared + private > num_pages:
        raise ValueError(f"pool of {num_pages} pages cannot hold {n_shared + private} pages")
    perm = permutation(num_pages, seed ^ 0x5A5A5A5A)
    pt = np.full((B, max_pages), -1, dtype=np.int32)
    cursor = n_shared
    for b in range(B):
        k = min(need[b], n_shared)
        pt[b, :k] = perm[:k]
        m = need[b] - k
        if m > 0:
            pt[b, k:k + m] = perm[cursor:cursor + m]
            cursor += m
    return pt


def custom(name: str, B: int, Hq: int, Hkv: int, D: int, prefix_lens, suffix_lens, *, ps: int = 16,
           shared_len: int = 0, num_pages: Optional[int] = None, seed: int = 0, extra_cols: int = 0) -> Workload:
    prefix_lens = np.asarray(prefix_lens, dtype=np.int32)
    suffix_lens = np.asarray(suffix_lens, dtype=np.int32)
    need = sum(-(-(int(p) + int(s)) // ps) for p, s in zip(prefix_lens, suffix_lens))
    if num_pages is None:
        num_pages = max(8, 2 * need)
    pt = place_pages(prefix_lens, suffix_lens, ps, num_pages, shared_len, seed, extra_cols)
    return Workload(name, B, Hq, Hkv, D, ps, prefix_lens, suffix_lens, shared_len, num_pages, pt, seed)


def _round_down(x, m):
    return (np.asarray(x, dtype=np.int64) // m) * m


def config(name: str, seed: int = 0, free_hbm_bytes: Optional[int] = None) -> Workload:
    """The five agent-shaped workloads (c3 has an LRU and an RR variant).

    c1_tiny       4 agents, 8/2 heads, d64, prefix U[256,1024] on pages, suffix U[32,128], 512-page pool
    c2_llama3_8b  32 agents, 32/8 heads, d128, prefix U[8k,32k] on 512-token chunk boundaries, suffix U[256,2048]
    c3_lru        64 agents, 32/8, d128, histories H~U[16k,64k]; 4 agents fully evicted down to the
                  2048-token shared system prompt with suffix U[32k,64k]; 60 fully cached, suffix 256
    c3_rr         same histories; every agent recomputes an equal share of c3_lru's uncached tokens
                  (S_i = U_tot/64, remainder spread one token each), P_i = H_i - S_i (mid-page)
    c4_coding     16 agents, 64/8, d128, prefix U[128k,256k] on pages, suffix U[1024,4096], pool = 90 % of
                  free HBM (pass `free_hbm_bytes`; without it a pool of 4x the needed pages is used)
    c5_shared     128 agents, 32/8, d128, 4096-token prefix shared by all (same physical pages), then a
                  private history U[4k,16k] on pages, suffix U[128,1024]
    """
    s = seed * 1000003
    ps = 16
    if name == "c1_tiny":
        B, Hq, Hkv, D = 4, 8, 2, 64
        P = _round_down(uniform_ints(B, 256, 1024, s + 1), ps)
        S = uniform_ints(B, 32, 128, s + 2)
        return custom(name, B, Hq, Hkv, D, P, S, ps=ps, num_pages=512, seed=seed)
    if name == "c2_llama3_8b":
        B, Hq, Hkv, D = 32, 32, 8, 128
        P = _round_down(uniform_ints(B, 8192, 32768, s + 1), 512)
        S = uniform_ints(B, 256, 2048, s + 2)
        return custom(name, B, Hq, Hkv, D, P, S, ps=ps, seed=seed)
    if name in ("c3_lru", "c3_rr"):
        B, Hq, Hkv, D = 64, 32, 8, 128
        shared = 2048
        H = _round_down(uniform_ints(B, 16384, 65536, s + 1), ps)
        evicted = set(int(i) for i in permutation(B, s + 3)[:4])
        S_lru = np.where(np.isin(np.arange(B), list(evicted)),
                         uniform_ints(B, 32768, 65536, s + 2), 256)
        P_lru = np.where(np.isin(np.arange(B), list(evicted)), shared, H)
        if name == "c3_lru":
            return custom(name, B, Hq, Hkv, D, P_lru, S_lru, ps=ps, shared_len=shared, seed=seed)
        u_tot = int(S_lru.sum())
        S = np.full(B, u_tot // B, dtype=np.int64)
        S[: u_tot % B] += 1
        P = H - S
        return custom(name, B, Hq, Hkv, D, P, S, ps=ps, shared_len=shared, seed=seed)
    if name == "c4_coding":
        B, Hq, Hkv, D = 16, 64, 8, 128
        P = _round_down(uniform_ints(B, 131072, 262144, s + 1), ps)
        S = uniform_ints(B, 1024, 4096, s + 2)
        need = sum(-(-(int(p) + int(q)) // ps) for p, q in zip(P, S))
        page_pair_bytes = 2 * ps * Hkv * D * 2
        if free_hbm_bytes is not None:
            num_pages = int(0.9 * free_hbm_bytes) // page_pair_bytes
        else:
            num_pages = 4 * need
        return custom(name, B, Hq, Hkv, D, P, S, ps=ps, num_pages=num_pages, seed=seed)
    if name == "c5_shared":
        B, Hq, Hkv, D = 128, 32, 8, 128
        shared = 4096
        Hp = _round_down(uniform_ints(B, 4096, 16384, s + 1), ps)
        S = uniform_ints(B, 128, 1024, s + 2)
        return custom(name, B, Hq, Hkv, D, shared + Hp, S, ps=ps, shared_len=shared, seed=seed)
    raise KeyError(name)


CONFIGS = ("c1_tiny", "c2_llama3_8b", "c3_lru", "c3_rr", "c4_coding", "c5_shared")

# Decode batches: the agents of an extend workload one step later -- each agent's history after its
# extend (P + S cached tokens) plus one new token (suffix 1), same heads, same shared prefix.
DECODE_CONFIGS = ("c2_decode", "c4_decode", "c5_decode")
_DECODE_BASE = {"c2_decode": "c2_llama3_8b", "c4_decode": "c4_coding", "c5_decode": "c5_shared"}


def decode_config(name: str, seed: int = 0, free_hbm_bytes: Optional[int] = None) -> Workload:
    """c2_decode: 32 agents, 32/8 heads, d128, keys = c2's P + S + 1 (~9k-35k)
    c4_decode: 16 agents, 64/8 heads, d128, keys = c4's P + S + 1 (~130k-265k), pool as c4_coding
    c5_decode: 128 agents, 32/8 heads, d128, keys = c5's P + S + 1, the 4096-token prefix shared by all"""
    base = config(_DECODE_BASE[name], seed, free_hbm_bytes)
    P = np.asarray(base.prefix_lens, dtype=np.int64) + np.asarray(base.suffix_lens, dtype=np.int64)
    num_pages = base.num_pages if name == "c4_decode" else None
    return custom(name, base.B, base.Hq, base.Hkv, base.D, P, np.ones(base.B, dtype=np.int64), ps=base.ps,
                  shared_len=base.shared_len, num_pages=num_pages, seed=seed)


# --------------------------------------------------------------------------- CPU tensors

def cpu_rows(wl: Workload, tensor: int, head0: int, head_count: int, row_agent=None, row_pos=None,
             nthreads: int = 0) -> np.ndarray:
    if row_agent is None:
        row_agent, row_pos = wl.row_agent_pos()
    row_agent = np.ascontiguousarray(row_agent, dtype=np.int32)
    row_pos = np.ascontiguousarray(row_pos, dtype=np.int64)
    n = len(row_pos)
    out = np.empty((n, head_count, wl.D), dtype=np.uint16)
    if n:
        cpu_lib().rrs_fill_rows(_ptr(out), _ptr(row_agent), _ptr(row_pos), n, head0, head_count, wl.D,
                                tensor, wl.seed & _U64, wl.shared_len, nthreads or (os.cpu_count() or 1))
    return out


def cpu_tensors(wl: Workload, pool_fill: int = BF16_NAN) -> Dict[str, np.ndarray]:
    """All inputs as bf16 bit patterns (uint16) on the host.

    k_pool/v_pool hold the cached prefix of every agent; every other slot holds
    `pool_fill` (a NaN by default, so a kernel that reads a slot it should not
    see poisons its output).
    """
    q = cpu_rows(wl, TENSOR_Q, 0, wl.Hq)
    k_new = cpu_rows(wl, TENSOR_K, 0, wl.Hkv)
    v_new = cpu_rows(wl, TENSOR_V, 0, wl.Hkv)
    shape = (wl.num_pages, wl.ps, wl.Hkv, wl.D)
    k_pool = np.full(shape, pool_fill, dtype=np.uint16)
    v_pool = np.full(shape, pool_fill, dtype=np.uint16)
    pt = np.ascontiguousarray(wl.page_table, dtype=np.int32)
    pl = np.ascontiguousarray(wl.prefix_lens, dtype=np.int32)
    cpu_lib().rrs_fill_pool_prefix(_ptr(k_pool), _ptr(v_pool), _ptr(pt), _ptr(pl), wl.B, wl.max_pages, wl.ps,
                                   wl.Hkv, wl.D, wl.seed & _U64, wl.shared_len, os.cpu_count() or 1)
    return dict(q=q, k_new=k_new, v_new=v_new, k_pool=k_pool, v_pool=v_pool)


def agent_kv(wl: Workload, b: int, n_pos: int, head: int, nthreads: int = 0):
    """Agent b's logical K and V for positions 0..n_pos-1 of KV head `head`: two [n_pos, D] uint16 arrays.

    Built from the generator by logical position only (never from a pool), so a
    page-indexing mistake anywhere else cannot leak into it.
    """
    agent = np.full(n_pos, b, dtype=np.int32)
    pos = np.arange(n_pos, dtype=np.int64)
    k = cpu_rows(wl, TENSOR_K, head, 1, agent, pos, nthreads)[:, 0, :]
    v = cpu_rows(wl, TENSOR_V, head, 1, agent, pos, nthreads)[:, 0, :]
    return k, v


def q_rows(wl: Workload, b: int, positions, nthreads: int = 0) -> np.ndarray:
    """q of agent b at the given absolute positions: [n, Hq, D] uint16."""
    positions = np.asarray(positions, dtype=np.int64)
    agent = np.full(len(positions), b, dtype=np.int32)
    return cpu_rows(wl, TENSOR_Q, 0, wl.Hq, agent, positions, nthreads)


def bf16_to_f64(a: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns."""
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------- GPU tensors

def gpu_tensors(wl: Workload, device="cuda", pool_fill: int = BF16_NAN, stream=None):
    """All inputs as torch bf16 tensors on `device`, values generated on the GPU.

    Bit-identical to cpu_tensors(wl).  Returns a dict with q, k_new, v_new,
    k_pool, v_pool (bf16) and page_table, prefix_lens, suffix_lens (int32).
    """
    import torch
    lib = cuda_lib()
    dev = torch.device(device)
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    sp = st.cuda_stream
    agent, pos = wl.row_agent_pos()
    t_agent = torch.from_numpy(agent.astype(np.int32)).to(dev)
    t_pos = torch.from_numpy(pos.astype(np.int64)).to(dev)
    T = wl.T

    def rows(tensor, heads):
        out = torch.empty((T, heads, wl.D), dtype=torch.bfloat16, device=dev)
        rc = lib.rrs_cuda_fill_rows(out.data_ptr(), t_agent.data_ptr(), t_pos.data_ptr(), T, 0, heads, wl.D,
                                    tensor, wl.seed & _U64, wl.shared_len, sp)
        if rc:
            raise RuntimeError(f"rrs_cuda_fill_rows failed: {rc}")
        return out

    q = rows(TENSOR_Q, wl.Hq)
    k_new = rows(TENSOR_K, wl.Hkv)
    v_new = rows(TENSOR_V, wl.Hkv)
    fill = np.array([pool_fill], dtype=np.uint16).view(np.int16)[0]
    shape = (wl.num_pages, wl.ps, wl.Hkv, wl.D)
    k_pool = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    v_pool = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    k_pool.view(torch.int16).fill_(int(fill))
    v_pool.view(torch.int16).fill_(int(fill))
    # one entry per (agent, prefix page); shared pages listed once (agent 0)
    ids, ag, p0, pe = [], [], [], []
    n_shared_pages = wl.shared_len // wl.ps
    for b in range(wl.B):
        P = int(wl.prefix_lens[b])
        first = 0 if b == 0 else min(n_shared_pages, -(-P // wl.ps))
        for pg in range(first, -(-P // wl.ps)):
            ids.append(int(wl.page_table[b, pg]))
            ag.append(b)
            p0.append(pg * wl.ps)
            pe.append(P)
    n_list = len(ids)
    if n_list:
        t_ids = torch.tensor(ids, dtype=torch.int32, device=dev)
        t_ag = torch.tensor(ag, dtype=torch.int32, device=dev)
        t_p0 = torch.tensor(p0, dtype=torch.int64, device=dev)
        t_pe = torch.tensor(pe, dtype=torch.int64, device=dev)
        for pool, tensor in ((k_pool, TENSOR_K), (v_pool, TENSOR_V)):
            rc = lib.rrs_cuda_fill_pool(pool.data_ptr(), t_ids.data_ptr(), t_ag.data_ptr(), t_p0.data_ptr(),
                                        t_pe.data_ptr(), n_list, wl.ps, wl.Hkv, wl.D, tensor, wl.seed & _U64,
                                        wl.shared_len, sp)
            if rc:
                raise RuntimeError(f"rrs_cuda_fill_pool failed: {rc}")
    return dict(q=q, k_new=k_new, v_new=v_new, k_pool=k_pool, v_pool=v_pool,
                page_table=torch.from_numpy(np.ascontiguousarray(wl.page_table)).to(dev),
                prefix_lens=torch.from_numpy(wl.prefix_lens.astype(np.int32)).to(dev),
                suffix_lens=torch.from_numpy(wl.suffix_lens.astype(np.int32)).to(dev))

"""Parity at the five workloads' full sizes, and on the LRU / RR-Evict pair drawn from the eviction-policy
generator, in the launch configuration bench.py times.

Attention: seeded sample of suffix rows (every sampled agent's first and last
row, a window of consecutive rows covering two whole Q tiles of the agent with
the longest prefix -- of each of 8 sampled agents on c4, whose key ranges are
the deepest -- and random rows up to an fp64 flop budget), all heads of each,
against the oracle computed from logically generated K/V -- never from the
GPU pool, so a page-indexing mistake cannot cancel out.

Append: every suffix slot, gathered back through the page table, equals its
k_new / v_new row bit for bit; every other slot of the pool keeps its content
(per-slot checksums before and after).
"""
import math
import os
import sys

import numpy as np
import pytest

import synth
from parity import check_close, oracle_sampled, sample_rows, to_f64

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402  (the workload definitions bench.py times)

pytestmark = pytest.mark.gpu

CONFIGS = ["c2_llama3_8b", "c3_lru", "c3_rr", "c5_shared", "c4_coding", "c3g_lru", "c3g_rr"]


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


def _slot_checksums(pool, chunk_slots=1 << 17):
    """int64 weighted sum of every token slot's bf16 bits: [num_pages * ps]."""
    import torch
    flat = pool.view(pool.shape[0] * pool.shape[1], -1).view(torch.int16)
    w = torch.arange(1, flat.shape[1] + 1, device=pool.device, dtype=torch.int64)
    out = torch.empty(flat.shape[0], dtype=torch.int64, device=pool.device)
    for s in range(0, flat.shape[0], chunk_slots):
        e = min(flat.shape[0], s + chunk_slots)
        out[s:e] = (flat[s:e].to(torch.int64) * w).sum(dim=1)
    return out


def _suffix_slots(wl):
    agent, pos = wl.row_agent_pos()
    pages = wl.page_table[agent, pos // wl.ps].astype(np.int64)
    return pages * wl.ps + pos % wl.ps


@pytest.mark.parametrize("name", CONFIGS)
def test_full_size_config(rr, name):
    import torch
    torch.cuda.empty_cache()
    free = torch.cuda.mem_get_info()[0]
    wl = bench.workload(synth, name, free_hbm_bytes=free if name == "c4_coding" else None)
    g = synth.gpu_tensors(wl, "cuda")
    before_k = _slot_checksums(g["k_pool"])
    before_v = _slot_checksums(g["v_pool"])

    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"])
    assert rr.device_error() == 0, rr.last_error()

    # ---- append: gather-back of every suffix slot, bit-exact
    slots = torch.from_numpy(_suffix_slots(wl)).cuda()
    for pool, new in ((g["k_pool"], g["k_new"]), (g["v_pool"], g["v_new"])):
        flat = pool.view(pool.shape[0] * pool.shape[1], wl.Hkv, wl.D)
        got = flat[slots].view(torch.int16)
        assert torch.equal(got, new.view(torch.int16)), f"{name}: appended rows differ"
    # ---- append: nothing else changed
    mask = torch.ones(wl.num_pages * wl.ps, dtype=torch.bool, device="cuda")
    mask[slots] = False
    assert torch.equal(_slot_checksums(g["k_pool"])[mask], before_k[mask]), f"{name}: k_pool changed off-suffix"
    assert torch.equal(_slot_checksums(g["v_pool"])[mask], before_v[mask]), f"{name}: v_pool changed off-suffix"
    del before_k, before_v, mask

    # ---- attention: sampled rows vs the oracle
    # c4 has the deepest key ranges (128k-256k): 8 agents, each with a whole work unit of consecutive rows
    deep = name == "c4_coding"
    rows = sample_rows(wl, flop_budget=2.5e11, seed=1, max_agents=8 if deep else 12, window_every_agent=deep)
    ref = oracle_sampled(wl, rows, 1.0 / math.sqrt(wl.D))
    cu = wl.cu
    got_rows, ref_rows = [], []
    for b, rs in rows.items():
        idx = torch.from_numpy(cu[b] + rs).cuda()
        got_rows.append(to_f64(out[idx]))
        ref_rows.append(ref[b])
    stats = check_close(np.concatenate(got_rows), np.concatenate(ref_rows), name)
    n_rows = sum(len(r) for r in rows.values())
    print(f"{name}: {n_rows} rows of {len(rows)} agents x {wl.Hq} heads checked ({stats['n']} elements in the "
          f"mean), max {stats['max']:.2e} mean {stats['mean']:.2e} p99.9 {stats['p999']:.2e}")
    del g, out
    torch.cuda.empty_cache()

"""The seeded input generator: determinism, published reference values, distribution, placement."""
import numpy as np
import pytest

import synth


def test_splitmix64_published_outputs():
    # SplitMix64 started from state 0: its first two outputs are the widely
    # published reference values of the generator (Steele, Lea, Flood 2014).
    w = synth.stream(2, 0)
    assert int(w[0]) == 0xE220A8397B1DCDAF
    assert int(w[1]) == 0x6E789E6AA1B965F4


def test_values_are_standard_normal_like():
    wl = synth.custom("t", 2, 4, 2, 64, [300, 0], [200, 100], seed=3)
    q = synth.bf16_to_f64(synth.cpu_tensors(wl)["q"]).ravel()
    assert abs(q.mean()) < 0.02
    assert abs(q.std() - 1.0) < 0.02
    assert np.all(np.abs(q) <= 6.0)


def test_values_depend_on_logical_coordinates_only():
    # same logical rows under two different page placements -> identical pool contents by position
    a = synth.custom("a", 2, 4, 2, 64, [64, 48], [10, 20], seed=5, num_pages=40)
    b = synth.custom("b", 2, 4, 2, 64, [64, 48], [10, 20], seed=5, num_pages=64)
    ta, tb = synth.cpu_tensors(a), synth.cpu_tensors(b)
    assert not np.array_equal(a.page_table, b.page_table) or a.num_pages != b.num_pages
    for b_ in range(2):
        for pos in range(int(a.prefix_lens[b_])):
            pa = a.page_table[b_, pos // 16]
            pb = b.page_table[b_, pos // 16]
            np.testing.assert_array_equal(ta["k_pool"][pa, pos % 16], tb["k_pool"][pb, pos % 16])
            np.testing.assert_array_equal(ta["v_pool"][pa, pos % 16], tb["v_pool"][pb, pos % 16])
    np.testing.assert_array_equal(ta["q"], tb["q"])


def test_agent_kv_matches_pool_prefix():
    wl = synth.custom("t", 3, 8, 2, 64, [80, 33, 0], [5, 7, 9], seed=11, shared_len=32)
    t = synth.cpu_tensors(wl)
    for b in range(wl.B):
        P = int(wl.prefix_lens[b])
        for g in range(wl.Hkv):
            k, v = synth.agent_kv(wl, b, P, g)
            for pos in range(P):
                page = wl.page_table[b, pos // 16]
                np.testing.assert_array_equal(k[pos], t["k_pool"][page, pos % 16, g])
                np.testing.assert_array_equal(v[pos], t["v_pool"][page, pos % 16, g])


def test_shared_prefix_pages_are_common():
    wl = synth.custom("t", 4, 4, 1, 64, [64, 80, 96, 48], [3, 3, 3, 3], shared_len=48, seed=2)
    for b in range(1, 4):
        np.testing.assert_array_equal(wl.page_table[b, :3], wl.page_table[0, :3])
    used = [int(x) for b in range(4) for x in wl.page_table[b, 3:] if x >= 0]
    assert len(used) == len(set(used))
    assert not set(used) & set(int(x) for x in wl.page_table[0, :3])


def test_page_placement_is_distinct_and_in_range():
    for name in ("c1_tiny", "c2_llama3_8b", "c5_shared"):
        wl = synth.config(name)
        n_shared = wl.shared_len // wl.ps
        pages = wl.page_table[:, n_shared:]
        live = pages[pages >= 0]
        assert live.min() >= 0 and live.max() < wl.num_pages
        assert len(np.unique(live)) == len(live)
        for b in range(wl.B):
            need = -(-(int(wl.prefix_lens[b]) + int(wl.suffix_lens[b])) // wl.ps)
            assert np.all(wl.page_table[b, :need] >= 0)
            assert np.all(wl.page_table[b, need:] == -1)


def test_config_shapes_follow_their_recipes():
    c1 = synth.config("c1_tiny")
    assert (c1.B, c1.Hq, c1.Hkv, c1.D, c1.num_pages) == (4, 8, 2, 64, 512)
    assert np.all(c1.prefix_lens % 16 == 0) and np.all((c1.prefix_lens >= 256) & (c1.prefix_lens <= 1024))
    assert np.all((c1.suffix_lens >= 32) & (c1.suffix_lens <= 128))
    c2 = synth.config("c2_llama3_8b")
    assert np.all(c2.prefix_lens % 512 == 0) and np.all((c2.prefix_lens >= 8192) & (c2.prefix_lens <= 32768))
    lru, rr = synth.config("c3_lru"), synth.config("c3_rr")
    assert lru.T == rr.T                                       # same total uncached tokens
    assert (lru.suffix_lens > 256).sum() == 4                  # four agents fully evicted
    assert np.all(lru.prefix_lens[lru.suffix_lens > 256] == 2048)
    assert rr.suffix_lens.max() - rr.suffix_lens.min() <= 1    # equal tail chunks
    assert 2000 <= rr.suffix_lens.min() and rr.suffix_lens.max() <= 4096
    ev = lru.suffix_lens > 256
    # RR keeps every history: cached prefix + recomputed tail = the same history the LRU agents cached
    np.testing.assert_array_equal((rr.prefix_lens + rr.suffix_lens)[~ev], lru.prefix_lens[~ev])
    c5 = synth.config("c5_shared")
    assert np.all(c5.page_table[:, :256] == c5.page_table[0, :256])
    c4 = synth.config("c4_coding")
    assert c4.G == 8 and np.all((c4.prefix_lens >= 131072) & (c4.prefix_lens <= 262144))


def test_manifest_fixes_the_inputs(tmp_path):
    """The manifest names everything the inputs depend on: the same config and seed give the same hash,
    another seed (another page placement) or another config a different one; written to JSON it reads back."""
    import json
    a = synth.config("c2_llama3_8b", seed=0).manifest()
    assert a == synth.config("c2_llama3_8b", seed=0).manifest()
    assert a["sha256"] != synth.config("c2_llama3_8b", seed=1).manifest()["sha256"]
    assert a["sha256"] != synth.config("c3_rr", seed=0).manifest()["sha256"]
    assert a["T"] == sum(a["suffix_lens"]) and len(a["prefix_lens"]) == a["B"] == 32
    wl = synth.custom("m", 2, 8, 2, 64, [16, 0], [5, 7], seed=3)
    path = tmp_path / "m.json"
    h = wl.write_manifest(str(path))
    back = json.loads(path.read_text())
    assert back["sha256"] == h and back["prefix_lens"] == [16, 0] and back["suffix_lens"] == [5, 7]


def test_manifest_hash_covers_seed_and_shapes():
    """Batches with the same lengths and page table but another value seed or head shape hash differently."""
    base = synth.custom("h", 2, 8, 2, 128, [64, 0], [10, 20], seed=3)
    h0 = base.manifest()["sha256"]
    variants = [
        synth.Workload(**{**base.__dict__, "seed": 4}),
        synth.Workload(**{**base.__dict__, "D": 64}),
        synth.Workload(**{**base.__dict__, "Hq": 16}),
        synth.Workload(**{**base.__dict__, "Hkv": 1}),
        synth.Workload(**{**base.__dict__, "num_pages": base.num_pages + 1}),
        synth.Workload(**{**base.__dict__, "shared_len": 16}),
    ]
    for v in variants:
        assert np.array_equal(v.page_table, base.page_table)
        assert v.manifest()["sha256"] != h0

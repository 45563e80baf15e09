"""Host logic of bench.py's stored ncu records (CPU only).

A recorded DRAM-traffic figure is reported only while it belongs to the code being timed: the source
hash ignores comments, blank lines and indentation but changes with any code line of the kernel's
files (the schedule's included, since its unit order sets the traffic), and a record is taken only for
the hash and the whole workload it was captured on.
"""
import json
import os
import shutil
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _tree(tmp_path):
    src = os.path.join(ROOT, "paper_2609_32278_gb300", "csrc")
    dst = tmp_path / "paper_2609_32278_gb300" / "csrc"
    shutil.copytree(src, dst, ignore=shutil.ignore_patterns("*.o", "*.so"))
    (tmp_path / "profiles").mkdir()
    return dst


def test_hash_ignores_comments_and_tracks_code(tmp_path, monkeypatch):
    csrc = _tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h_attn = bench.kernel_source_hash()
    h_dec = bench.kernel_source_hash(bench.DECODE_SOURCES)
    assert h_attn == bench.kernel_source_hash(bench.ATTN_SOURCES) and h_attn != h_dec
    f = csrc / "extend_attn.cu"
    f.write_text("// a new comment line\n\n" + f.read_text().replace("\n", "   // trailing comment\n", 1))
    assert bench.kernel_source_hash() == h_attn
    s = csrc / "sched.cu"
    s.write_text(s.read_text() + "\nstatic int unused_marker = 1;\n")
    assert bench.kernel_source_hash() != h_attn                       # the schedule is part of the attention's
    assert bench.kernel_source_hash(bench.DECODE_SOURCES) != h_dec    # and of the decode kernel's sources
    d = csrc / "decode_attn.cu"
    h_attn2 = bench.kernel_source_hash()
    d.write_text(d.read_text() + "\nstatic int other_marker = 2;\n")
    assert bench.kernel_source_hash() == h_attn2                      # decode code is not the attention's


def test_record_taken_only_for_its_hash(tmp_path, monkeypatch):
    _tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h = bench.kernel_source_hash()
    recs = {"c4_coding": {"dram_bytes_per_launch": 123, "slice": "c4_coding[:2]"},
            "c4_coding[:2]": {"dram_bytes_per_launch": 17}}
    rec = {"kernel_source_hash": h, "records": recs}
    (tmp_path / "profiles" / "extend_attn_traffic.json").write_text(json.dumps(rec))
    got, raw = bench.load_traffic(h)
    assert got == recs and raw == rec
    assert bench.traffic_for("c4_coding", h) == 123
    assert bench.traffic_for("c4_coding[:2]", h) == 17
    assert bench.traffic_for("c2_llama3_8b", h) is None                        # not recorded
    got, raw = bench.load_traffic("0" * 16)
    assert got is None and raw == rec
    assert bench.traffic_for("c4_coding", "0" * 16) is None                   # recorded on other code
    assert bench.load_traffic(h, "decode_attn_traffic.json") == (None, None)   # no such record


def test_both_arms_name_the_same_config():
    """The reference arm builds the coding-agent batch without a GPU (pool size unknown); the config both
    arms report leaves the pool size out, so it is the same."""
    import synth
    a = synth.config("c4_coding", seed=0, free_hbm_bytes=250 * 2 ** 30)
    b = synth.config("c4_coding", seed=0)
    assert a.num_pages != b.num_pages
    assert bench.config_dict(a, 1) == bench.config_dict(b, 1)



def test_policy_pair_workloads():
    """The generator-drawn skew pair (bench legs c3g_lru / c3g_rr): same agents, the shared system prompt on
    common pages, whole-history recomputes under LRU against short tails under RR-Evict, valid page tables."""
    import numpy as np
    import synth
    a = bench.workload(synth, "c3g_lru")
    b = bench.workload(synth, "c3g_rr")
    assert a.B == b.B > 32 and a.shared_len == b.shared_len == 2048
    assert (a.Hq, a.Hkv, a.D) == (b.Hq, b.Hkv, b.D) == (32, 8, 128)
    assert a.suffix_lens.max() > 8 * b.suffix_lens.max()
    assert np.all(a.prefix_lens >= 2048) and np.all(b.prefix_lens >= 2048)
    # every agent's first 128 logical pages are the shared ones
    assert np.all(a.page_table[:, :128] == a.page_table[0, :128])
    import paper_2609_32278_gb300 as rr
    if os.path.exists(rr._SO):
        for w in (a, b):
            assert rr.validate_page_table(w.page_table, w.prefix_lens, w.suffix_lens, w.num_pages, w.ps) == 0


def test_tensor_peak_follows_the_timed_loop_length():
    """A timed loop of a second or more runs in the power-capped regime of the sustained GEMM figure; a shorter
    one is held to the burst figure.  Both are the measured numbers, never a mix."""
    peaks = dict(hbm=6685.8, bf16=1881.8, bf16_sus=1741.7, src="measured")
    p, kind = bench.tensor_peak(peaks, 190.0)          # c2: 20 steps of ~9.5 ms
    assert p == 1881.8 and "burst" in kind
    p, kind = bench.tensor_peak(peaks, 20 * 213.0)     # c4: 20 steps of ~213 ms
    assert p == 1741.7 and "sustained" in kind
    p, _ = bench.tensor_peak(peaks, bench.SUSTAINED_AFTER_MS)
    assert p == 1741.7
    fb = dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")
    p, kind = bench.tensor_peak(fb, 5000.0)
    assert p == 1700.0 and kind.startswith("fallback")

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
    rec = {"kernel_source_hash": h, "workload": "c2_llama3_8b", "dram_bytes_per_launch": 123}
    (tmp_path / "profiles" / "extend_attn_traffic.json").write_text(json.dumps(rec))
    got, raw = bench.load_traffic(h)
    assert got == rec and raw == rec
    got, raw = bench.load_traffic("0" * 16)
    assert got is None and raw == rec
    assert bench.load_traffic(h, "decode_attn_traffic.json") == (None, None)   # no such record


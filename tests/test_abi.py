"""The C ABI library on a machine without a GPU: it loads, exports every declared symbol, and its
host-only entry points (page-table validation, version, error strings) behave."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rr.h")


def _rr():
    import paper_2609_32278_gb300 as rr
    if not os.path.exists(rr._SO):
        pytest.skip("librr.so not built (run __graft_entry__.build())")
    return rr


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rr_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    import paper_2609_32278_gb300 as rr
    assert declared_symbols() == sorted(rr.EXPORTS)


def test_library_exports_every_declared_symbol():
    rr = _rr()
    lib = ctypes.CDLL(rr._SO)
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_version_and_empty_error():
    rr = _rr()
    assert "sm_103a" in rr.version()
    assert rr.last_error() == ""


def _table(prefix, suffix, ps, seed=0, shared=0, num_pages=None):
    import synth
    wl = synth.custom("v", len(prefix), 1, 1, 64, prefix, suffix, ps=ps, shared_len=shared, seed=seed,
                      num_pages=num_pages)
    return wl


def test_validate_accepts_generated_tables():
    rr = _rr()
    import synth
    for name in ("c1_tiny", "c2_llama3_8b", "c3_rr", "c5_shared"):
        wl = synth.config(name)
        assert rr.validate_page_table(wl.page_table, wl.prefix_lens, wl.suffix_lens, wl.num_pages, wl.ps) == 0, \
            rr.last_error()


def test_validate_rejects_out_of_pool_page():
    rr = _rr()
    wl = _table([40, 10], [5, 30], 16)
    pt = wl.page_table.copy()
    pt[1, 2] = wl.num_pages
    assert rr.validate_page_table(pt, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16) == rr.RR_ERR_OOB
    pt[1, 2] = -1
    assert rr.validate_page_table(pt, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16) == rr.RR_ERR_OOB


def test_validate_rejects_shared_suffix_page():
    rr = _rr()
    wl = _table([40, 10], [5, 30], 16)
    pt = wl.page_table.copy()
    pt[1, 1] = pt[0, 2]           # agent 1's suffix page is agent 0's suffix page
    assert rr.validate_page_table(pt, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16) == rr.RR_ERR_OVERLAP
    pt = wl.page_table.copy()
    pt[1, 0] = pt[0, 2]           # agent 1 (whose first page holds suffix positions) writes into agent 0's page
    assert rr.validate_page_table(pt, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16) == rr.RR_ERR_OVERLAP


def test_validate_allows_shared_prefix_pages():
    rr = _rr()
    wl = _table([64, 80, 48], [10, 20, 16], 16, shared=48)
    assert rr.validate_page_table(wl.page_table, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16) == 0


def test_validate_rejects_bad_lengths():
    rr = _rr()
    wl = _table([40, 10], [5, 30], 16)
    assert rr.validate_page_table(wl.page_table, wl.prefix_lens, wl.suffix_lens, wl.num_pages, 16,
                                  total_tokens=34) == rr.RR_ERR_LENS
    assert "total_tokens" in rr.last_error()
    bad = np.array([40, -1], dtype=np.int32)
    assert rr.validate_page_table(wl.page_table, wl.prefix_lens, bad, wl.num_pages, 16) == rr.RR_ERR_LENS

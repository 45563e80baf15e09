"""Seeded random batches through the append, the extend attention, the one-launch step and decode, plain and
with a rotary table, and batches with a shared prefix through the extend cascade and the shared-prefix decode,
against the fp64 oracle.

Each case draws its own shape -- head dim 64 or 128, 1-8 KV heads, GQA group 1-16, page size 8-128 -- and a
batch of 1-9 agents whose cached prefixes may be empty, end mid-page or run to a few thousand keys, and whose
suffixes may be empty, one token or a few hundred, so that the cases between them cross every Q-tile and
KV-tile boundary the kernels have, split-K and unsplit schedules, and the append's partly owned last pages.
The append is compared bit-exact on the whole pool (untouched slots included), the attention within the parity
bar; the one-launch step must reproduce the two calls bit for bit; decode runs on the appended pools with one
new query per agent.  The seeds are fixed, so a failure names its case.
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, to_f64

pytestmark = pytest.mark.gpu

N_CASES = 64


def draw_case(i):
    rng = np.random.default_rng(7000 + i)
    D = int(rng.choice([64, 128]))
    while True:
        Hkv = int(rng.choice([1, 2, 4, 8]))
        G = int(rng.choice([1, 2, 4, 8, 16]))
        if G * Hkv <= 32:
            break
    ps = int(rng.choice([8, 16, 32, 64, 128]))
    B = int(rng.integers(1, 10))
    kind_p = rng.random(B)
    P = np.where(kind_p < 0.2, 0, np.where(kind_p < 0.6, rng.integers(1, 300, B), rng.integers(300, 2000, B)))
    kind_s = rng.random(B)
    S = np.where(kind_s < 0.1, 0, np.where(kind_s < 0.2, 1, rng.integers(2, 220, B)))
    if S.sum() == 0:
        S[0] = 5
    return dict(name=f"fuzz{i}", B=B, Hq=G * Hkv, Hkv=Hkv, D=D, ps=ps, P=P.astype(np.int64), S=S.astype(np.int64),
                seed=100 + i)


CASES = [draw_case(i) for i in range(N_CASES)]


def case_id(c):
    return f"{c['name']}-D{c['D']}-Hkv{c['Hkv']}-G{c['Hq'] // c['Hkv']}-ps{c['ps']}-B{c['B']}"


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    return m


@pytest.mark.parametrize("case", CASES, ids=[case_id(c) for c in CASES])
def test_random_batch(rr, case):
    import torch
    wl = synth.custom(case["name"], case["B"], case["Hq"], case["Hkv"], case["D"], case["P"], case["S"],
                      ps=case["ps"], seed=case["seed"])
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    g2 = {k: v.clone() for k, v in g.items()}

    # append + attention, two calls
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"])
    torch.cuda.synchronize()
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                              wl.prefix_lens, wl.suffix_lens)
    np.testing.assert_array_equal(bf16_bits(g["k_pool"]), kp)
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)
    ref = oracle.extend_attention(host["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                  scale=1.0 / math.sqrt(wl.D))
    check_close(to_f64(out), ref, f"{case_id(case)} extend")

    # the one-launch step on fresh copies of the same inputs: the same pools and output, bit for bit
    out2 = rr.extend_step(g2["q"], g2["k_new"], g2["v_new"], g2["k_pool"], g2["v_pool"], g2["page_table"],
                          g2["prefix_lens"], g2["suffix_lens"])
    torch.cuda.synchronize()
    assert rr.device_error() == 0, rr.last_error()
    np.testing.assert_array_equal(bf16_bits(g2["k_pool"]), kp)
    np.testing.assert_array_equal(bf16_bits(out2), bf16_bits(out))

    # decode on the appended pool: one new query per agent over all its keys (agents with at least one key)
    L = wl.prefix_lens.astype(np.int64) + wl.suffix_lens.astype(np.int64)
    if (L >= 1).all():
        rng = np.random.default_rng(case["seed"])
        qd_bits = np.ascontiguousarray(oracle.round_bf16(rng.standard_normal((wl.B, wl.Hq, wl.D))))  # bf16 bits
        qd_t = torch.from_numpy(qd_bits.view(np.int16).copy()).view(torch.bfloat16).cuda()
        kv_lens = torch.tensor(L, dtype=torch.int32, device="cuda")
        outd = rr.decode_attention(qd_t, g["k_pool"], g["v_pool"], g["page_table"], kv_lens)
        torch.cuda.synchronize()
        assert rr.device_error() == 0, rr.last_error()
        refd = oracle.decode_attention(qd_bits, kp, vp, wl.page_table, L.astype(np.int32),
                                       scale=1.0 / math.sqrt(wl.D))
        check_close(to_f64(outd), refd, f"{case_id(case)} decode")


BASE = 500000.0


@pytest.mark.parametrize("case", CASES[::2], ids=[case_id(c) for c in CASES[::2]])
def test_random_batch_rotary(rr, case):
    """The same batches with q and k_new taken un-rotated (rotary table, base 5e5): the rotated append (V bit-exact;
    K is checked against its error bound in the rotary tests) and attention against the oracle's rotation, and
    the one-launch rotary step bit-identical to the two calls."""
    import torch
    wl = synth.custom(case["name"], case["B"], case["Hq"], case["Hkv"], case["D"], case["P"], case["S"],
                      ps=case["ps"], seed=case["seed"])
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    g2 = {k: v.clone() for k, v in g.items()}
    table = rr.rope_table(int((wl.prefix_lens.astype(np.int64) + wl.suffix_lens).max()) + 1, wl.D, BASE)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"], rope=table)
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"], rope=table)
    torch.cuda.synchronize()
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append_rope(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                                   wl.prefix_lens, wl.suffix_lens, BASE)
    np.testing.assert_array_equal(bf16_bits(g["v_pool"]), vp)
    ref = oracle.extend_attention_rope(host["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens, BASE,
                                       scale=1.0 / math.sqrt(wl.D))
    check_close(to_f64(out), ref, f"{case_id(case)} rotary extend")
    out2 = rr.extend_step(g2["q"], g2["k_new"], g2["v_new"], g2["k_pool"], g2["v_pool"], g2["page_table"],
                          g2["prefix_lens"], g2["suffix_lens"], rope=table)
    torch.cuda.synchronize()
    assert rr.device_error() == 0, rr.last_error()
    np.testing.assert_array_equal(bf16_bits(g2["k_pool"]), bf16_bits(g["k_pool"]))
    np.testing.assert_array_equal(bf16_bits(out2), bf16_bits(out))


def draw_shared_case(i):
    rng = np.random.default_rng(9000 + i)
    D = int(rng.choice([64, 128]))
    while True:
        Hkv = int(rng.choice([1, 2, 4, 8]))
        G = int(rng.choice([1, 2, 4, 8, 16]))
        if G * Hkv <= 32:
            break
    ps = int(rng.choice([8, 16, 32, 64, 128]))
    B = int(rng.integers(1, 12))
    shared = int(rng.choice([128, 256, 384, 512]))
    P = shared + np.where(rng.random(B) < 0.25, 0, rng.integers(1, 1500, B))
    kind_s = rng.random(B)
    S = np.where(kind_s < 0.1, 0, np.where(kind_s < 0.2, 1, rng.integers(2, 220, B)))
    if S.sum() == 0:
        S[0] = 3
    return dict(name=f"fuzzsh{i}", B=B, Hq=G * Hkv, Hkv=Hkv, D=D, ps=ps, P=P.astype(np.int64),
                S=S.astype(np.int64), shared=shared, seed=300 + i)


SHARED_CASES = [draw_shared_case(i) for i in range(24)]


@pytest.mark.parametrize("case", SHARED_CASES, ids=[case_id(c) + f"-sh{c['shared']}" for c in SHARED_CASES])
def test_random_batch_shared_prefix(rr, case):
    """Batches whose agents share their first shared_len positions (the same pages): the extend cascade
    (rr_extend_attention_shared) and the shared-prefix decode (rr_decode_attention_shared) against the oracle."""
    import torch
    wl = synth.custom(case["name"], case["B"], case["Hq"], case["Hkv"], case["D"], case["P"], case["S"],
                      ps=case["ps"], shared_len=case["shared"], seed=case["seed"])
    host = synth.cpu_tensors(wl)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    out = rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                              g["suffix_lens"], shared_len=case["shared"])
    torch.cuda.synchronize()
    assert rr.device_error() == 0, rr.last_error()
    kp, vp = oracle.kv_append(host["k_new"], host["v_new"], host["k_pool"], host["v_pool"], wl.page_table,
                              wl.prefix_lens, wl.suffix_lens)
    ref = oracle.extend_attention(host["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                  scale=1.0 / math.sqrt(wl.D))
    check_close(to_f64(out), ref, f"{case_id(case)} cascade")
    L = wl.prefix_lens.astype(np.int64) + wl.suffix_lens.astype(np.int64)
    if (L > case["shared"]).all():  # every agent needs a private key for the shared-prefix decode
        rng = np.random.default_rng(case["seed"])
        qd_bits = np.ascontiguousarray(oracle.round_bf16(rng.standard_normal((wl.B, wl.Hq, wl.D))))
        qd_t = torch.from_numpy(qd_bits.view(np.int16).copy()).view(torch.bfloat16).cuda()
        kv_lens = torch.tensor(L, dtype=torch.int32, device="cuda")
        outd = rr.decode_attention(qd_t, g["k_pool"], g["v_pool"], g["page_table"], kv_lens,
                                   shared_len=case["shared"])
        torch.cuda.synchronize()
        assert rr.device_error() == 0, rr.last_error()
        refd = oracle.decode_attention(qd_bits, kp, vp, wl.page_table, L.astype(np.int32),
                                       scale=1.0 / math.sqrt(wl.D))
        check_close(to_f64(outd), refd, f"{case_id(case)} shared decode")

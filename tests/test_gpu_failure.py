"""The bounded-wait failure path of the attention kernels, provoked without a GPU fault.

rr_set_wait_limit shortens the budget of the kernels' pipeline waits (every wait of the decode kernel,
the stage watcher's in the extend kernel, the one-launch step's grid barrier), and with it how long one try may suspend the thread, to a
few hundred clock cycles, far below a tile's load time, so the first such wait runs out.  Each such call must end with RR_ERR_TIMEOUT in the device error word -- every role leaves its
loop, copies and tensor-core operations in flight are drained, tensor memory is freed -- and the context
must stay usable: with the default budget restored, the same call returns, bit for bit, what it returned
before the timeout, and that matches the oracle.  Covered: the extend kernel (unsplit and split-K
batches), the one-launch extend step and the decode kernel.  Every agent has cached keys, so no row
sees only a handful of keys (those rows' bf16 error margin is tested elsewhere; here the subject is
the recovery).
"""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import bf16_bits, check_close, to_f64

pytestmark = pytest.mark.gpu

SHORT = 400  # clock cycles


@pytest.fixture(scope="module")
def rr():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32278_gb300 as m
    m.lib()
    yield m
    m.set_wait_limit(0)


def reference(wl):
    t = synth.cpu_tensors(wl)
    kp, vp = oracle.kv_append(t["k_new"], t["v_new"], t["k_pool"], t["v_pool"], wl.page_table, wl.prefix_lens,
                              wl.suffix_lens)
    return oracle.extend_attention(t["q"], kp, vp, wl.page_table, wl.prefix_lens, wl.suffix_lens,
                                   scale=1.0 / math.sqrt(wl.D))


def timed_out(rr, call):
    rr.set_wait_limit(SHORT)
    try:
        call()
        code = rr.device_error()
    finally:
        rr.set_wait_limit(0)
    return code


@pytest.mark.parametrize("case", [
    ("unsplit", 6, [3000, 700, 16, 1500, 2048, 64], [129, 70, 200, 300, 64, 33]),
    ("split", 1, [20000], [50]),
], ids=lambda c: c[0])
def test_extend_wait_runs_out_and_the_context_recovers(rr, case):
    name, B, P, S = case
    wl = synth.custom(f"timeout_{name}", B, 8, 2, 128, P, S, seed=41)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    assert rr.device_error() == 0

    def attend():
        return rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                   g["suffix_lens"])

    before = bf16_bits(attend()).copy()
    assert rr.device_error() == 0
    assert timed_out(rr, attend) == rr.RR_ERR_TIMEOUT
    out = attend()
    assert rr.device_error() == 0
    assert np.array_equal(bf16_bits(out), before)
    check_close(to_f64(out), reference(wl), f"after timeout ({name})")


def test_fused_step_wait_runs_out_and_the_context_recovers(rr):
    wl = synth.custom("timeout_fused", 3, 8, 2, 128, [37, 2000, 16], [129, 70, 300], seed=42)
    g = synth.gpu_tensors(wl, "cuda")

    def step():
        return rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                              g["prefix_lens"], g["suffix_lens"])

    before = bf16_bits(step()).copy()
    assert rr.device_error() == 0
    assert timed_out(rr, step) == rr.RR_ERR_TIMEOUT
    out = step()
    assert rr.device_error() == 0
    assert np.array_equal(bf16_bits(out), before)
    check_close(to_f64(out), reference(wl), "fused step after timeout")


def test_decode_wait_runs_out_and_the_context_recovers(rr):
    import torch
    L = np.array([9000, 300, 4000], dtype=np.int64)
    wl = synth.custom("timeout_decode", 3, 8, 2, 128, L - 1, np.ones(3, dtype=np.int64), seed=43)
    g = synth.gpu_tensors(wl, "cuda")
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    kv = (g["prefix_lens"] + 1).to(torch.int32)

    def decode():
        return rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv)

    before = bf16_bits(decode()).copy()
    assert rr.device_error() == 0
    assert timed_out(rr, decode) == rr.RR_ERR_TIMEOUT
    out = decode()
    assert rr.device_error() == 0
    assert np.array_equal(bf16_bits(out), before)
    check_close(to_f64(out), reference(wl), "decode after timeout")

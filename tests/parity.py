"""Shared helpers of the GPU parity tests: tolerance check, row sampling, oracle on sampled rows."""
from __future__ import annotations

import math

import numpy as np

import oracle
import synth

# Attention parity bar (bf16 inputs, fp32 accumulation): fp64 oracle vs the bf16 output.
MAX_ABS = 1e-2
MEAN_ABS = 1e-3
# Where |ref| >= 2 the output's own rounding to bf16 (half a unit in the last place: 2^-7 on [2, 4),
# 2^-6 on [4, 8)) takes most or all of MAX_ABS, so there the bar is MAX_ABS plus that half unit.
ROUNDING_FROM = 2.0


def max_abs_bar(ref: np.ndarray) -> np.ndarray:
    """Per-element bound on |got - ref|: MAX_ABS, plus half a bf16 unit in the last place of ref where
    |ref| >= ROUNDING_FROM (bf16 keeps 8 significant bits, so on [2^e, 2^(e+1)) half a unit is 2^(e-8))."""
    a = np.abs(np.asarray(ref, dtype=np.float64))
    _, e = np.frexp(np.maximum(a, ROUNDING_FROM))  # a = m 2^e with m in [0.5, 1): floor(log2 a) = e - 1
    return MAX_ABS + np.where(a >= ROUNDING_FROM, np.ldexp(1.0, e - 9), 0.0)


def bf16_bits(t) -> np.ndarray:
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def to_f64(t) -> np.ndarray:
    return synth.bf16_to_f64(bf16_bits(t))


def _ordered(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> integers in the order of their values (one step = one unit in the last place)."""
    b = bits.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def check_close(got: np.ndarray, ref: np.ndarray, what: str = "") -> dict:
    """Parity of a bf16 GPU output (as float64) with the fp64 oracle: every |err| within max_abs_bar(ref)
    and the mean |err| within MEAN_ABS, plus the 99.9th percentile |err| and the distance in bf16 units in
    the last place to the oracle rounded to bf16 (round to nearest even, once), printed on one line."""
    err = np.abs(got - ref)
    stats = dict(n=int(err.size), max=float(err.max()) if err.size else 0.0,
                 mean=float(err.mean()) if err.size else 0.0,
                 p999=float(np.quantile(err, 0.999)) if err.size else 0.0,
                 max_over_bar=float((err / max_abs_bar(ref)).max()) if err.size else 0.0)
    assert np.isfinite(got).all(), f"{what}: non-finite outputs"
    if err.size:
        ulp = np.abs(_ordered(oracle.round_bf16(got)) - _ordered(oracle.round_bf16(ref)))
        stats.update(ulp_max=int(ulp.max()), ulp_le1=float(np.mean(ulp <= 1)), ulp_eq0=float(np.mean(ulp == 0)))
    print(f"parity {what}: {stats}")
    assert stats["max_over_bar"] <= 1.0 and stats["mean"] <= MEAN_ABS, f"{what}: {stats}"
    return stats


def sample_rows(wl: synth.Workload, flop_budget: float = 4e11, seed: int = 0, max_agents: int = 12,
                window_every_agent: bool = False):
    """Suffix rows (agent, row) to check on a full-size config, within an fp64 flop budget.

    Agents: all of them if there are at most `max_agents`, else the agents with
    the longest prefix, the longest suffix and the shortest context plus seeded
    random others (regenerating each sampled agent's K/V on the CPU is the
    expensive part).  Rows: each sampled agent's first and last row; one window
    of consecutive rows (every row position of two Q tiles, i.e. one whole work
    unit, and a few of the next) of the agent with the longest prefix, or of
    every sampled agent with `window_every_agent`; then seeded random rows
    while the budget lasts (the windows are taken whatever they cost).
    """
    rng = np.random.default_rng(seed)
    cost = lambda b: 4.0 * wl.D * wl.Hq * (int(wl.prefix_lens[b]) + int(wl.suffix_lens[b]))
    live_all = [b for b in range(wl.B) if wl.suffix_lens[b] > 0]
    if len(live_all) > max_agents:
        must = {max(live_all, key=lambda b: int(wl.prefix_lens[b])),
                max(live_all, key=lambda b: int(wl.suffix_lens[b])),
                min(live_all, key=lambda b: int(wl.prefix_lens[b]) + int(wl.suffix_lens[b]))}
        rest = [b for b in live_all if b not in must]
        extra = rng.choice(rest, size=max(0, max_agents - len(must)), replace=False)
        live = sorted(must | set(int(x) for x in extra))
    else:
        live = live_all
    picked = {b: set() for b in live}
    spent = 0.0
    for b in live:
        S = int(wl.suffix_lens[b])
        for i in {0, S - 1}:
            picked[b].add(i)
            spent += cost(b)
    if live:
        win_agents = live if window_every_agent else [max(live, key=lambda b: int(wl.prefix_lens[b]))]
        for bw in win_agents:
            window = min(int(wl.suffix_lens[bw]), 2 * 128 // wl.G + 5)
            for i in range(window):
                if i not in picked[bw]:
                    picked[bw].add(i)
                    spent += cost(bw)
    tries = 0
    while spent < flop_budget and live and tries < 100000:
        tries += 1
        b = int(rng.choice(live))
        i = int(rng.integers(0, int(wl.suffix_lens[b])))
        if i in picked[b]:
            continue
        picked[b].add(i)
        spent += cost(b)
    return {b: np.array(sorted(v), dtype=np.int64) for b, v in picked.items() if v}


def oracle_sampled(wl: synth.Workload, rows_by_agent, scale=None, nthreads=0):
    """fp64 oracle on sampled rows from logically generated K/V (never from a pool).

    Returns {agent: array [n_rows, Hq, D]} for the rows in rows_by_agent.
    """
    if scale is None:
        scale = 1.0 / math.sqrt(wl.D)
    out = {}
    for b, rows in rows_by_agent.items():
        P = int(wl.prefix_lens[b])
        pos = P + rows
        L = int(pos.max()) + 1
        qr = synth.q_rows(wl, b, pos, nthreads)
        res = np.zeros((len(rows), wl.Hq, wl.D))
        for g in range(wl.Hkv):
            K, V = synth.agent_kv(wl, b, L, g, nthreads)
            res[:, g * wl.G:(g + 1) * wl.G] = oracle.attention_rows(qr[:, g * wl.G:(g + 1) * wl.G], pos, K, V,
                                                                   scale, nthreads)
        out[b] = res
    return out

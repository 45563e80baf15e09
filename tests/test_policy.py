"""The eviction policies (Sec. 3): Algorithm 1 step by step on hand-built trees, LRU's recency-synchronised
behaviour, and the analytical model of Sec. 3.3 (Eq. 1-3) -- closed forms and the policies run on it."""
import json
import os

import pytest

from paper_2609_32278_gb300 import policy as pol

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _cache(lengths, capacity=None, page=16, times=None, shared=0):
    c = pol.RadixCache(capacity or (sum(sum(x) for x in lengths) + shared), page)
    if shared:
        c.add_shared_prefix(shared)
    for a, segs in enumerate(lengths):
        c.add_agent(a)
        for s in segs:
            c.insert(a, s, float(times[a]) if times else float(a))
    return c


# ---------------------------------------------------------------- Algorithm 1

def test_rr_visits_agents_round_robin():
    c = _cache([[4096], [4096], [4096]])
    freed = pol.evict_rr(c, 3 * 1024, chunk=1024)
    assert freed == 3 * 1024
    assert [c.private_len(a) for a in range(3)] == [3072, 3072, 3072]


def test_rr_stops_once_demand_is_met():
    c = _cache([[4096], [4096], [4096]])
    freed = pol.evict_rr(c, 1500, chunk=1024)
    # first agent: a full chunk; second: the rest of the demand rounded up to a page (476 -> 480)
    assert [c.private_len(a) for a in range(3)] == [3072, 4096 - 480, 4096]
    assert freed == 1024 + 480


def test_rr_partial_leaf_stays_next_candidate():
    c = _cache([[3000]])
    pol.evict_rr(c, 1024, chunk=1024)
    leaf = c.tail[0]
    assert leaf.length == 3000 - 1024 and leaf.owner == 0
    pol.evict_rr(c, 1024, chunk=1024)
    assert c.tail[0] is leaf and leaf.length == 3000 - 2048


def test_rr_exposes_parent_only_when_leaf_is_gone():
    c = _cache([[512, 300]])           # two private nodes: a parent and a leaf of 300
    first, second = c.path(0)
    pol.evict_rr(c, 100, chunk=1024)   # partial: the leaf shrinks, parent untouched
    assert second.length == 300 - 112 and first.length == 512
    pol.evict_rr(c, 188, chunk=1024)   # the rest of the leaf; now the parent is the tail leaf
    assert c.tail[0] is first and first.length == 512
    pol.evict_rr(c, 1024, chunk=1024)
    assert c.private_len(0) == 0


def test_rr_skips_active_agents_and_rechecks():
    c = _cache([[2048], [2048], [2048]])
    c.set_active(1, True)
    pol.evict_rr(c, 4 * 1024, chunk=1024)
    assert c.private_len(1) == 2048
    assert c.private_len(0) == 0 and c.private_len(2) == 0


def test_rr_drops_trajectories_with_nothing_left():
    c = _cache([[256], [4096]])
    freed = pol.evict_rr(c, 2048, chunk=1024)
    assert c.private_len(0) == 0 and c.private_len(1) == 4096 - (2048 - 256)
    assert freed == 2048


def test_rr_never_evicts_shared_prefix_while_private_state_remains():
    c = _cache([[1024], [1024]], shared=2048)
    pol.evict_rr(c, 1024, chunk=1024)
    assert c.shared.length == 2048 and c.shared.parent is c.root


def test_rr_queue_starts_with_least_recent_agent():
    c = _cache([[4096], [4096], [4096]], times=[5, 1, 3])
    pol.evict_rr(c, 1024, chunk=1024)
    assert [c.private_len(a) for a in range(3)] == [4096, 3072, 4096]


# ---------------------------------------------------------------- LRU behaviour

def test_lru_concentrates_on_the_oldest_agent_under_recency_synchronisation():
    # every agent's nodes were refreshed together (match), so its private nodes share one recency
    c = _cache([[512] * 8, [512] * 8, [512] * 8], times=[3, 1, 2])
    for a, t in enumerate([3, 1, 2]):
        c.match(a, float(t))
    pol.evict_lru(c, 4096)
    assert [c.private_len(a) for a in range(3)] == [4096, 0, 4096]


def test_lru_frees_whole_nodes_leaf_first():
    c = _cache([[1000, 700]])
    pol.evict_lru(c, 100)
    assert c.private_len(0) == 1000                 # the whole 700-token leaf went
    pol.evict_lru(c, 1)
    assert c.private_len(0) == 0


def test_completion_signal_frees_private_state_only():
    c = _cache([[1000, 700], [300]], shared=128)
    assert c.complete(0) == 1700
    assert c.private_len(1) == 300 and c.shared.length == 128


def test_tiered_drains_old_tier_round_robin_first():
    c = _cache([[2048], [2048], [2048], [2048]], times=[0.1, 0.2, 5.1, 5.2])
    pol.evict_tiered(c, 2048, chunk=1024, tier_width=1.0)
    assert [c.private_len(a) for a in range(4)] == [1024, 1024, 2048, 2048]


# ---------------------------------------------------------------- Sec. 3.3 analytical model

def test_eq1_eq2_eq3_closed_forms_golden():
    with open(os.path.join(GOLDEN, "rr_analysis.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        assert pol.rr_regime(c["n"], c["a"], c["m"]) == c["in_regime"]
        if c["in_regime"]:
            h, q = pol.rr_hit_miss(c["n"], c["a"], c["m"])
            assert h == pytest.approx(c["h"], abs=1e-12)
            assert q == pytest.approx(c["q"], abs=1e-12)
            lru, rr = pol.recompute_cost_distribution(c["n"], c["a"], c["m"])
            mean_lru = sum(v * p for v, p in lru.items())
            mean_rr = sum(v * p for v, p in rr.items())
            assert mean_lru == pytest.approx(c["q"]) and mean_rr == pytest.approx(c["q"])   # same mean, Sec. 3.3


@pytest.mark.parametrize("n,na,m", [(40, 8, 30.0), (64, 16, 48.0), (20, 2, 11.0)])
def test_policies_realise_eq2_and_eq3_on_the_homogeneous_model(n, na, m):
    U = 16384
    chunk = 1024
    h, q = pol.rr_hit_miss(n, na / n, m)
    rr = pol.homogeneous_eviction(n, na, m, U, "rr", chunk)
    lru = pol.homogeneous_eviction(n, na, m, U, "lru", chunk)
    ns = n - na
    # RR: every idle agent recomputes about q of its prefix (within one chunk)
    for x in rr.values():
        assert abs(x - q * U) <= chunk
    # LRU: n - m idle agents lose everything, the others nothing (Eq. 3's two-point law)
    full = sum(1 for x in lru.values() if x == U)
    none = sum(1 for x in lru.values() if x == 0)
    assert full + none == ns and full == round(n - m)
    # both recompute the same total: mean miss q (Sec. 3.3)
    assert sum(rr.values()) / (ns * U) == pytest.approx(q, abs=chunk / U)
    assert sum(lru.values()) / (ns * U) == pytest.approx(q, abs=1e-12)
    # and the worst case drops from a full prefix to ~q of one
    assert max(lru.values()) == U and max(rr.values()) <= q * U + chunk


def test_replay_rr_cuts_the_uncached_tail():
    import random
    rnd = random.Random(0)
    traces = []
    for a in range(24):
        turns = 6
        traces.append(pol.AgentTrace(new_tokens=[rnd.randint(2000, 6000) if k == 0 else rnd.randint(200, 800)
                                                 for k in range(turns)],
                                     output_tokens=[rnd.randint(50, 300) for _ in range(turns)],
                                     gaps=[rnd.uniform(0.5, 3.0) for _ in range(turns)],
                                     start=rnd.uniform(0, 2.0)))
    cap = 24 * 5500     # active contexts fit, all live histories do not (Eq. 1's regime)
    res = {}
    for p in ("lru", "rr"):
        reqs = pol.replay(traces, cap, p, shared_prompt=512, chunk=1024)
        unc = sorted(r.uncached for r in reqs if r.turn > 0)
        res[p] = (unc[int(0.99 * (len(unc) - 1))], sum(unc) / len(unc), max(unc))
        assert all(r.cached <= r.prompt_len for r in reqs)
    assert res["rr"][0] < res["lru"][0]      # P99 uncached tokens (Sec. 4 metric)
    assert res["rr"][2] < res["lru"][2]

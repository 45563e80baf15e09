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


# ----------------------------------------------------------------------------- replay with admission, metrics

def test_synthetic_traces_are_seeded_and_in_range():
    a = pol.synthetic_traces(30, "conversational", seed=3)
    b = pol.synthetic_traces(30, "conversational", seed=3)
    c = pol.synthetic_traces(30, "conversational", seed=4)
    assert [t.new_tokens for t in a] == [t.new_tokens for t in b]
    assert [t.new_tokens for t in a] != [t.new_tokens for t in c]
    for t in a:
        assert 8 <= len(t.new_tokens) <= 30 and len(t.output_tokens) == len(t.gaps) == len(t.new_tokens)
        assert 300 <= t.new_tokens[0] <= 1500 and all(100 <= x <= 1500 for x in t.new_tokens[1:])
        assert all(0.5 <= g <= 90.0 for g in t.gaps)
    for t in pol.synthetic_traces(10, "coding", seed=0):
        assert 15 <= len(t.new_tokens) <= 60 and all(300 <= x <= 6000 for x in t.new_tokens[1:])
    with pytest.raises(ValueError):
        pol.synthetic_traces(1, "chat")


def test_replay_never_admits_more_than_the_concurrency():
    traces = pol.synthetic_traces(40, "coding", seed=1)
    conc = 7
    reqs = pol.replay(traces, 10 ** 9, "lru", concurrency=conc)
    first, last = {}, {}
    for r in reqs:
        first.setdefault(r.agent, r.time)
        last[r.agent] = r.time
    assert len(first) == 40                            # every agent is eventually admitted
    for r in reqs:
        live = sum(1 for a in first if first[a] <= r.time <= last[a])
        assert live <= conc
    # with unbounded capacity every turn after the first reuses the whole previous context
    by_agent = {}
    for r in reqs:
        by_agent.setdefault(r.agent, []).append(r)
    for a, rs in by_agent.items():
        for k in range(1, len(rs)):
            assert rs[k].cached == rs[k - 1].prompt_len + traces[a].output_tokens[k - 1]


def test_percentile_is_nearest_rank():
    v = list(range(1, 101))
    assert pol.percentile(v, 99) == 99 and pol.percentile(v, 50) == 50 and pol.percentile(v, 100) == 100
    assert pol.percentile([5], 99) == 5 and pol.percentile([3, 1, 2], 0) == 1


def test_extend_batches_group_by_arrival_window():
    def req(agent, t, cached, uncached):
        return pol.Request(agent, 0, t, cached + uncached, cached)

    reqs = [req(0, 0.00, 60, 40), req(1, 0.03, 0, 50), req(2, 0.06, 60, 10), req(3, 0.04, 0, 90),
            req(4, 0.20, 30, 0), req(5, 0.21, 55, 5)]
    got = pol.extend_batches(reqs, window=0.05)
    # [0.00, 0.05]: requests 0, 1, 3 (in arrival order); then 2 alone; 4 has nothing uncached; then 5
    assert [b[0] for b in got] == [[0, 1, 3], [2], [5]]
    assert got[0][1] == [60, 0, 0] and got[0][2] == [40, 50, 90]
    assert got[2][1] == [55] and got[2][2] == [5]
    flat = sorted(i for b in got for i in b[0])
    assert flat == [i for i, r in enumerate(reqs) if r.uncached > 0]


def test_snapshot_lengths_take_each_agents_next_request():
    # Request(agent, turn, time, prompt_len, cached)
    reqs = [pol.Request(0, 0, 0.0, 100, 0), pol.Request(1, 0, 1.0, 200, 0), pol.Request(0, 1, 2.0, 300, 150),
            pol.Request(1, 1, 3.0, 400, 20), pol.Request(0, 2, 4.0, 500, 500), pol.Request(1, 2, 5.0, 600, 90)]
    # the median request arrives at t = 3.0: agent 0's next is its turn 2, agent 1's its turn 1
    P, S = pol.snapshot_lengths(reqs, 0.5)
    assert P == [500, 20] and S == [0, 380]


def test_snapshot_pair_shows_the_two_recompute_shapes():
    """The generator-drawn skew pair: under LRU a few agents recompute their whole history (long suffixes
    over the shared prompt alone), under RR-Evict every agent recomputes a shorter tail (Eq. 3)."""
    traces = pol.synthetic_traces(64, "coding", seed=0)
    finals = sorted(sum(t.new_tokens) + sum(t.output_tokens) for t in traces)
    cap = int(0.5 * sum(finals))
    res = {}
    for label, policy, cs in (("lru", "lru", False), ("rr", "rr", True)):
        reqs = pol.replay(traces, cap, policy, shared_prompt=2048, chunk=1024, completion_signals=cs,
                          concurrency=64)
        res[label] = pol.snapshot_lengths(reqs, 0.5)
    (Pl, Sl), (Pr, Sr) = res["lru"], res["rr"]
    assert len(Sl) == len(Sr) > 32
    assert max(Sl) > 8 * max(Sr) and sum(Sl) > sum(Sr)
    assert min(Pl) == 2048 and min(Pr) >= 2048   # the shared system prompt is never evicted


def test_summarize_reports_the_sec4_metrics():
    reqs = [pol.Request(0, k, float(k), 100 + k, 100 - k) for k in range(50)]
    s = pol.summarize(reqs, times=[1e-3 * r.uncached for r in reqs])
    assert s["requests"] == 50 and s["uncached_max"] == 2 * 49
    assert s["uncached_p99"] == pol.percentile([2 * k for k in range(50)], 99)
    assert s["ttft_attn_max_ms"] == pytest.approx(98.0)


def test_rr_cuts_the_tail_on_the_synthetic_conversational_replay():
    """Sec. 4's comparison on the seeded conversational traces, at a capacity inside Eq. 1's regime."""
    traces = pol.synthetic_traces(222, "conversational", seed=0)
    finals = sorted(sum(t.new_tokens) + sum(t.output_tokens) for t in traces)
    cap = int(0.4 * sum(finals[-40:]))
    p99 = {}
    for label, policy, cs in (("lru", "lru", False), ("lru+cs", "lru", True), ("rr", "rr", True)):
        reqs = pol.replay(traces, cap, policy, shared_prompt=2048, chunk=1024, completion_signals=cs,
                          concurrency=40)
        p99[label] = pol.summarize(reqs)["uncached_p99"]
    assert p99["rr"] < p99["lru+cs"] < p99["lru"]

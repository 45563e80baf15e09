"""Prefix-cache eviction policies over a radix tree -- the host side of RR-Evict.

This is the part of the system the paper changes (Sec. 3): it decides how much
of each agent's history survives in the KV pool, and therefore the cached
prefix P_b and uncached suffix S_b of every returning agent that the GPU
kernels then process.  Pure Python on the CPU; not on the GPU path.

Model
-----
* A ``RadixCache`` holds, per agent, a path from the root: an optional node
  shared by every agent (a common system prompt) followed by a chain of
  private nodes, one per insertion (turn).  Lengths are in tokens; the pool
  frees whole pages of ``page_size`` tokens.
* A node is *active* while an executing request references it (Sec. 3.1);
  active nodes are never evicted.  Eviction only ever removes a leaf, or a
  suffix of a leaf, so every agent keeps a contiguous cached prefix.
* ``match`` (a returning agent's prefix lookup) refreshes the last-access
  time of every node on the agent's surviving path at once -- the recency
  synchronisation of Sec. 1 / Sec. 3.1.

Policies
--------
* ``evict_lru``: eligible leaves in a heap ordered by last access; pop, free
  the whole node, push its parent when it becomes an eligible leaf (Sec. 3.1).
* ``evict_rr``: Algorithm 1 (Sec. 3.2).  Idle trajectories with an evictable
  suffix enter one queue; pop the front, skip it if it became active or has
  nothing left, free one tail chunk chosen by ``select_tail_chunk`` (a whole
  leaf or a suffix of it; a partly freed leaf stays the next candidate), push
  the trajectory back while it still has an evictable suffix; stop once the
  requested memory is freed or the queue is empty.
* ``evict_tiered``: recency tiering (Sec. 3.2, "Handling stale agent
  trajectories"): idle trajectories are grouped into tiers of last-access time,
  tiers are drained least recent first, round-robin inside a tier.  The paper
  describes but does not evaluate it.
* ``complete``: a completion signal frees the agent's unshared cache at once.

Readings where the paper is silent:
* queue order at the start of a reclamation: least recently accessed first,
  ties by agent id;
* SelectTailChunk frees min(chunk, leaf length, remaining demand rounded up to
  a page), and never less than a page unless the leaf is shorter;
* a node shared by several agents belongs to no trajectory; it is evicted by
  the LRU fallback only once nothing else can be freed.
"""
from __future__ import annotations

import dataclasses
import heapq
import itertools
from collections import deque
from typing import Dict, List, Optional

SHARED = -1


@dataclasses.dataclass(eq=False)
class Node:
    nid: int
    parent: Optional["Node"]
    length: int
    owner: int                    # agent id, or SHARED
    last_access: float = 0.0
    children: List["Node"] = dataclasses.field(default_factory=list)

    @property
    def is_leaf(self) -> bool:
        return not self.children


class RadixCache:
    """Token-level radix tree of agent histories over a pool of `capacity` tokens."""

    def __init__(self, capacity: int, page_size: int = 16):
        self.capacity = int(capacity)
        self.page_size = int(page_size)
        self._ids = itertools.count()
        self.root = Node(next(self._ids), None, 0, SHARED)
        self.used = 0
        self.shared: Optional[Node] = None
        self.tail: Dict[int, Node] = {}      # agent -> last node of its cached path (root if nothing cached)
        self.active: Dict[int, bool] = {}

    # ------------------------------------------------------------------ structure
    def add_shared_prefix(self, length: int, now: float = 0.0) -> Node:
        assert self.shared is None
        self.shared = Node(next(self._ids), self.root, int(length), SHARED, now)
        self.root.children.append(self.shared)
        self.used += int(length)
        return self.shared

    def add_agent(self, agent: int) -> None:
        base = self.shared if self.shared is not None else self.root
        self.tail[agent] = base
        self.active[agent] = False

    def path(self, agent: int) -> List[Node]:
        out = []
        n = self.tail[agent]
        while n is not None and n is not self.root:
            out.append(n)
            n = n.parent
        return out[::-1]

    def cached_len(self, agent: int) -> int:
        return sum(n.length for n in self.path(agent))

    def private_len(self, agent: int) -> int:
        return sum(n.length for n in self.path(agent) if n.owner == agent)

    @property
    def free(self) -> int:
        return self.capacity - self.used

    # ------------------------------------------------------------------ requests
    def match(self, agent: int, now: float) -> int:
        """Longest cached prefix of the agent's next prompt; refreshes recency along the path."""
        for n in self.path(agent):
            n.last_access = now
        return self.cached_len(agent)

    def insert(self, agent: int, n_tokens: int, now: float) -> Node:
        """Append n_tokens of this agent's context after its cached path (a new private leaf)."""
        if n_tokens > self.free:
            raise MemoryError(f"insert of {n_tokens} tokens with {self.free} free")
        parent = self.tail[agent]
        node = Node(next(self._ids), parent, int(n_tokens), agent, now)
        parent.children.append(node)
        self.tail[agent] = node
        self.used += int(n_tokens)
        return node

    def set_active(self, agent: int, active: bool) -> None:
        self.active[agent] = active

    def _node_active(self, node: Node) -> bool:
        if node.owner == SHARED:
            return any(self.active[a] for a in self.tail)
        return self.active.get(node.owner, False)

    def _remove(self, node: Node) -> None:
        node.parent.children.remove(node)
        for a, t in self.tail.items():
            if t is node:
                self.tail[a] = node.parent

    def _shrink(self, node: Node, tokens: int) -> int:
        tokens = min(tokens, node.length)
        node.length -= tokens
        self.used -= tokens
        if node.length == 0:
            self._remove(node)
        return tokens

    # ------------------------------------------------------------------ trajectories
    def evictable_leaf(self, agent: int) -> Optional[Node]:
        """The agent's private tail leaf if it is evictable now (idle, a leaf, private)."""
        if self.active.get(agent, False):
            return None
        t = self.tail[agent]
        if t is self.root or t.owner != agent or not t.is_leaf:
            return None
        return t

    def complete(self, agent: int) -> int:
        """Completion signal: free the agent's unshared cache now."""
        freed = 0
        while True:
            t = self.tail[agent]
            if t is self.root or t.owner != agent or not t.is_leaf:
                return freed
            freed += self._shrink(t, t.length)


def select_tail_chunk(cache: RadixCache, leaf: Node, demand: int, chunk: int) -> int:
    """Tokens to free from the tail of `leaf`: a whole leaf or a suffix of it (Sec. 3.2)."""
    ps = cache.page_size
    want = min(chunk, demand)
    want = -(-want // ps) * ps            # whole pages
    return max(1, min(leaf.length, want))


def _queue_order(cache: RadixCache, agents) -> List[int]:
    def key(a):
        path = cache.path(a)
        return (path[-1].last_access if path else 0.0, a)
    return sorted(agents, key=key)


def evict_rr(cache: RadixCache, M: int, chunk: int = 1024) -> int:
    """Algorithm 1: round-robin tail eviction over idle trajectories until M tokens are freed."""
    queue = deque(_queue_order(cache, [a for a in cache.tail if cache.evictable_leaf(a) is not None]))
    freed = 0
    while freed < M and queue:
        tau = queue.popleft()
        leaf = cache.evictable_leaf(tau)            # eligibility rechecked before every eviction
        if leaf is None:
            continue
        c = select_tail_chunk(cache, leaf, M - freed, chunk)
        freed += cache._shrink(leaf, c)
        if cache.evictable_leaf(tau) is not None:
            queue.append(tau)
    if freed < M:
        freed += _evict_shared_fallback(cache, M - freed)
    return freed


def evict_lru(cache: RadixCache, M: int) -> int:
    """Node-level LRU: min-heap of eligible leaves by last access; whole nodes are freed."""
    heap = []
    seen = set()

    def push(n: Node):
        if n is cache.root or not n.is_leaf or cache._node_active(n) or n.nid in seen:
            return
        seen.add(n.nid)
        heapq.heappush(heap, (n.last_access, n.nid, n))

    def walk(n: Node):
        for c in n.children:
            walk(c)
        push(n)

    walk(cache.root)
    freed = 0
    while freed < M and heap:
        _, _, n = heapq.heappop(heap)
        if n.parent is None or n not in n.parent.children or not n.is_leaf or cache._node_active(n):
            continue
        parent = n.parent
        freed += cache._shrink(n, n.length)
        if parent is not cache.root:
            push(parent)
    return freed


def evict_tiered(cache: RadixCache, M: int, chunk: int = 1024, tier_width: float = 1.0) -> int:
    """Recency tiering: LRU across tiers of last-access time, round-robin within a tier."""
    agents = [a for a in cache.tail if cache.evictable_leaf(a) is not None]
    tiers: Dict[int, List[int]] = {}
    for a in agents:
        t = cache.path(a)[-1].last_access
        tiers.setdefault(int(t // tier_width), []).append(a)
    freed = 0
    for k in sorted(tiers):
        if freed >= M:
            break
        queue = deque(_queue_order(cache, tiers[k]))
        while freed < M and queue:
            tau = queue.popleft()
            leaf = cache.evictable_leaf(tau)
            if leaf is None:
                continue
            freed += cache._shrink(leaf, select_tail_chunk(cache, leaf, M - freed, chunk))
            if cache.evictable_leaf(tau) is not None:
                queue.append(tau)
    if freed < M:
        freed += _evict_shared_fallback(cache, M - freed)
    return freed


def _evict_shared_fallback(cache: RadixCache, M: int) -> int:
    s = cache.shared
    if s is None or s.parent is None or not s.is_leaf or cache._node_active(s):
        return 0
    return cache._shrink(s, s.length)


def evict(cache: RadixCache, M: int, policy: str, chunk: int = 1024, tier_width: float = 1.0) -> int:
    if M <= 0:
        return 0
    if policy == "lru":
        return evict_lru(cache, M)
    if policy == "rr":
        return evict_rr(cache, M, chunk)
    if policy == "tiered":
        return evict_tiered(cache, M, chunk, tier_width)
    raise KeyError(policy)


# ---------------------------------------------------------------------- analytical model (Sec. 3.3)

def rr_regime(n: float, a: float, m: float) -> bool:
    """Eq. 1: distributing eviction over idle agents helps only when n*a < m < n."""
    return n * a < m < n


def rr_hit_miss(n: float, a: float, m: float):
    """Eq. 2: retained fraction h = (m - n a) / (n s) and miss q = 1 - h = (n - m) / (n s), s = 1 - a."""
    s = 1.0 - a
    h = (m - n * a) / (n * s)
    return h, 1.0 - h


def recompute_cost_distribution(n: float, a: float, m: float):
    """Eq. 3: normalised old-prefix recomputation of a uniformly chosen returning idle agent.

    LRU: 1 with probability q, else 0.  Ideal RR: q with probability 1.  Returns
    ({value: probability} for LRU, {value: probability} for RR).
    """
    _, q = rr_hit_miss(n, a, m)
    return {1.0: q, 0.0: 1.0 - q}, {q: 1.0}


# ---------------------------------------------------------------------- homogeneous experiment

def homogeneous_eviction(n: int, n_active: int, m_prefixes: float, prefix_tokens: int, policy: str,
                         chunk: int = 1024, page_size: int = 16, seed: int = 0):
    """Sec. 3.3's workload, run through the real policies.

    n agents with equal private prefixes of `prefix_tokens` and no sharing;
    `n_active` of them pinned (active), the rest idle with distinct last-access
    times; the pool holds `m_prefixes` prefixes.  Evicts down to capacity and
    returns {agent: tokens that agent must recompute on return}.
    """
    import random
    rnd = random.Random(seed)
    cap = int(round(m_prefixes * prefix_tokens))
    cache = RadixCache(n * prefix_tokens, page_size)
    agents = list(range(n))
    times = list(range(n))
    rnd.shuffle(times)
    for a in agents:
        cache.add_agent(a)
        cache.insert(a, prefix_tokens, float(times[a]))
    active = set(rnd.sample(agents, n_active))
    for a in agents:
        cache.set_active(a, a in active)
    cache.capacity = cap
    need = cache.used - cap
    evict(cache, need, policy, chunk)
    return {a: prefix_tokens - cache.private_len(a) for a in agents if a not in active}


# ---------------------------------------------------------------------- trace replay

@dataclasses.dataclass
class AgentTrace:
    """One agent's turns: new prompt tokens appended at each turn, output tokens, idle gap after it."""
    new_tokens: List[int]
    output_tokens: List[int]
    gaps: List[float]
    start: float = 0.0


@dataclasses.dataclass
class Request:
    agent: int
    turn: int
    time: float
    prompt_len: int
    cached: int

    @property
    def uncached(self) -> int:
        # Sec. 4: uncached tokens = prompt length - cached prefix length
        return self.prompt_len - self.cached


def replay(traces: List[AgentTrace], capacity: int, policy: str, shared_prompt: int = 0, chunk: int = 1024,
           page_size: int = 16, completion_signals: bool = True, tier_width: float = 1.0,
           service_time_per_token: float = 1e-4, concurrency: Optional[int] = None) -> List[Request]:
    """Replay agent traces against one prefix cache under `policy`; returns every request.

    Each turn: prefix match (refreshing recency), eviction of what the uncached
    part needs, insertion of prompt + output, an active period proportional to
    the uncached tokens, then the recorded idle gap.  A finished agent's unshared
    cache is released at once if `completion_signals`.

    `concurrency` caps the admitted agents (Sec. 4's replay: the agent slots are
    filled first, then a new agent is admitted only when a resident one exits;
    an admitted agent stays admitted while idle between turns).  None admits
    every trace at its start time.
    """
    cache = RadixCache(capacity, page_size)
    if shared_prompt:
        cache.add_shared_prefix(shared_prompt)
    events = []
    hist = {}
    waiting = deque()
    for a, tr in enumerate(traces):
        cache.add_agent(a)
        hist[a] = shared_prompt
        if concurrency is None or a < concurrency:
            heapq.heappush(events, (tr.start, 0, a, 0))      # (time, kind 0=arrive 1=finish, agent, turn)
        else:
            waiting.append(a)
    out: List[Request] = []
    while events:
        now, kind, a, k = heapq.heappop(events)
        tr = traces[a]
        if kind == 1:
            cache.set_active(a, False)
            if k + 1 < len(tr.new_tokens):
                heapq.heappush(events, (now + tr.gaps[k], 0, a, k + 1))
            else:
                if completion_signals:
                    cache.complete(a)
                if waiting:  # the slot passes to the next agent in line
                    heapq.heappush(events, (now, 0, waiting.popleft(), 0))
            continue
        prompt = hist[a] + tr.new_tokens[k]
        cached = cache.match(a, now)
        cached = min(cached, prompt)
        out.append(Request(a, k, now, prompt, cached))
        cache.set_active(a, True)
        need = (prompt - cached) + tr.output_tokens[k]
        if need > cache.free:
            evict(cache, need - cache.free, policy, chunk, tier_width)
        grow = min(need, cache.free)
        if grow > 0:
            cache.insert(a, grow, now)
        hist[a] = prompt + tr.output_tokens[k]
        busy = service_time_per_token * (prompt - cached + tr.output_tokens[k])
        heapq.heappush(events, (now + busy, 1, a, k))
    return out


# --------------------------------------------------------------------------- synthetic agent traces

def synthetic_traces(n_agents: int, kind: str = "conversational", seed: int = 0) -> List[AgentTrace]:
    """Seeded agent traces shaped like the paper's two workloads (Sec. 4), which are not available here.

    conversational -- customer-service agents (the tau^2-bench banking shape): 8-30 turns; a first
      user message of 300-1500 tokens, then per turn 100-1500 appended tokens (tool results or the
      user's reply); 30-400 output tokens; after a tool call a short gap (0.5-4 s), after a reply
      to the user a long pause (10-90 s) -- one turn in three waits for the user.
    coding -- software-engineering agents (the SWE-bench shape): 15-60 turns; a first message of
      1000-4000 tokens (issue + repository summary), then 300-6000 appended tokens per turn (file
      views, test logs); 50-800 output tokens; gaps of 1-20 s (tool and test execution).
    Agents start over the first 30 s.  Token counts are uniform on the ranges, gaps uniform on
    theirs; every number comes from one seeded generator, none from any dataset.
    """
    import random
    rnd = random.Random((seed * 1000003) ^ (0x5EED if kind == "coding" else 0xC0DE))
    out = []
    for _ in range(n_agents):
        if kind == "conversational":
            turns = rnd.randint(8, 30)
            new = [rnd.randint(300, 1500)] + [rnd.randint(100, 1500) for _ in range(turns - 1)]
            outs = [rnd.randint(30, 400) for _ in range(turns)]
            gaps = [rnd.uniform(10.0, 90.0) if rnd.random() < 1 / 3 else rnd.uniform(0.5, 4.0) for _ in range(turns)]
        elif kind == "coding":
            turns = rnd.randint(15, 60)
            new = [rnd.randint(1000, 4000)] + [rnd.randint(300, 6000) for _ in range(turns - 1)]
            outs = [rnd.randint(50, 800) for _ in range(turns)]
            gaps = [rnd.uniform(1.0, 20.0) for _ in range(turns)]
        else:
            raise ValueError(kind)
        out.append(AgentTrace(new_tokens=new, output_tokens=outs, gaps=gaps, start=rnd.uniform(0.0, 30.0)))
    return out


def percentile(values, p: float) -> float:
    """Nearest-rank percentile (p in [0, 100]) of a non-empty sequence."""
    v = sorted(values)
    k = max(0, min(len(v) - 1, int(-(-p * len(v) // 100)) - 1))
    return float(v[k])


def summarize(requests: List[Request], times=None) -> Dict[str, float]:
    """Sec. 4's per-request metrics: uncached prompt tokens (P50, P99, mean, max) and, given each request's
    measured extend time in seconds (`times[i]` for requests[i]; 0 for a request with nothing to extend),
    the attention part of its time to first token (P50, P99, mean, max)."""
    unc = [r.uncached for r in requests]
    res = {"requests": len(requests), "uncached_p50": percentile(unc, 50), "uncached_p99": percentile(unc, 99),
           "uncached_mean": sum(unc) / len(unc), "uncached_max": float(max(unc))}
    if times is not None:
        t = list(times)
        res.update({"ttft_attn_p50_ms": 1e3 * percentile(t, 50), "ttft_attn_p99_ms": 1e3 * percentile(t, 99),
                    "ttft_attn_mean_ms": 1e3 * sum(t) / len(t), "ttft_attn_max_ms": 1e3 * max(t)})
    return res


def extend_batches(requests: List[Request], window: float = 0.05):
    """The extend batches a prefill engine launches: requests in arrival order, each batch taking every
    request that arrives within `window` seconds of its first one (one scheduling tick).  Returns a list of
    (request indices, prefix_lens, suffix_lens); requests with nothing uncached are left out (no extend)."""
    order = sorted((i for i, r in enumerate(requests) if r.uncached > 0), key=lambda i: (requests[i].time, i))
    out = []
    k = 0
    while k < len(order):
        t0 = requests[order[k]].time
        j = k
        while j < len(order) and requests[order[j]].time - t0 <= window:
            j += 1
        idx = order[k:j]
        out.append((idx, [requests[i].cached for i in idx], [requests[i].uncached for i in idx]))
        k = j
    return out


def snapshot_lengths(requests: List[Request], quantile: float = 0.5):
    """(prefix_lens, suffix_lens) of the batch in which every agent returns at once: each agent's first
    request at or after the time by which `quantile` of all requests have arrived, in agent order.  The
    cached prefixes are what the policy left each agent at that moment, so the batch has the policy's
    (P, S) distribution (Sec. 3.3, Eq. 3)."""
    times = sorted(r.time for r in requests)
    t_star = times[min(len(times) - 1, int(len(times) * quantile))]
    first: Dict[int, Request] = {}
    for r in sorted(requests, key=lambda r: (r.time, r.agent)):
        if r.time >= t_star and r.agent not in first:
            first[r.agent] = r
    agents = sorted(first)
    return [first[a].cached for a in agents], [first[a].uncached for a in agents]

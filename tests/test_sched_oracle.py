"""CPU pins of the serving-order, finite-cache and pinned-layout oracles
(Sec. 7.1, Sec. 8, Thm 7), with planted mistakes in the cache simulator."""

from __future__ import annotations

import inspect
import itertools

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I

pytestmark = pytest.mark.timeout(300)


def _random_strings(rng, m, n, kmax, share=0.6):
    """Strings that share prefixes: each copies a prefix of an earlier one
    with probability ``share``, then adds distinct fresh-ish chunks."""
    out = []
    for i in range(m):
        if out and rng.random() < share:
            base = out[int(rng.integers(len(out)))]
            pre = list(base[:int(rng.integers(0, len(base) + 1))])
        else:
            pre = []
        k = int(rng.integers(0, kmax + 1))
        rest = [int(x) for x in rng.permutation(n) if int(x) not in pre][:max(0, k - len(pre))]
        out.append(pre + rest)
    return out


def test_cache_hand_example():
    """Strings ab, ac, ab, d (w = a:5 b:3 c:4 d:7) served in order.  Capacity 0
    caches nothing: 8 + 9 + 8 + 7 = 32.  Capacity 8: the first request fills
    the cache (a, b); the second hits a, pays c (4) and, as a and c do not fit
    with b, evicts b and leaves c uncached; the third hits a and pays b (3);
    the fourth pays d: 8 + 4 + 3 + 7 = 22.  Capacity 12 holds a, b, c: the third
    request hits both, total 19 = the trie weight 5 + 3 + 4 + 7."""
    w = np.array([5, 3, 4, 7])
    s = [[0, 1], [0, 2], [0, 1], [3]]
    assert O.radix_cache_costs(w, s, [0, 1, 2, 3], [0, 5, 8, 12, 10 ** 6]) == [32, 22, 22, 19, 19]
    assert O.trie_cost(w, s) == 19
    # in Thm 7's order (ab, ab, ac, d) one request's context (8) already suffices
    order = O.serve_order(s)
    assert order == [0, 2, 1, 3]
    assert O.radix_cache_cost(w, s, order, 8) == 19


def test_cache_recency_example():
    """Strings a, b, a, c, a (unit weights).  Capacity 2: a, b fill the cache,
    the second a hits and becomes the most recent, so c evicts b, and the last
    a hits: 3 paid.  Capacity 1 keeps only the latest string: 5 paid.
    Capacity 3 holds a, b, c: 3 paid."""
    w = np.ones(3, dtype=np.int64)
    s = [[0], [1], [0], [2], [0]]
    assert O.radix_cache_costs(w, s, [0, 1, 2, 3, 4], [0, 1, 2, 3]) == [5, 5, 3, 3]


def test_thm7_any_layout():
    """Thm 7: for ANY layout, serving in lexicographic order with capacity
    max_i w(string i) pays exactly the unbounded-cache cost (the trie weight)."""
    rng = np.random.default_rng(5)
    for trial in range(25):
        m = int(rng.integers(1, 30))
        n = int(rng.integers(3, 12))
        s = _random_strings(rng, m, n, 6)
        w = rng.integers(1, 50, size=n)
        order = O.serve_order(s)
        cap = max([sum(int(w[x]) for x in q) for q in s] + [0])
        trie = O.trie_cost(w, s)
        assert O.radix_cache_cost(w, s, order, cap) == trie
        assert O.radix_cache_cost(w, s, order, 10 ** 9) == trie


def test_capacity_limits_and_monotone():
    """Capacity 0 pays every string in full; a capacity holding the whole trie
    pays the trie weight in any order; cost never rises with capacity (LRU is
    a stack algorithm)."""
    rng = np.random.default_rng(9)
    for trial in range(15):
        m = int(rng.integers(1, 25))
        n = int(rng.integers(3, 10))
        s = _random_strings(rng, m, n, 5)
        w = rng.integers(1, 30, size=n)
        order = [int(x) for x in rng.permutation(m)]
        total = sum(int(w[x]) for q in s for x in q)
        trie = O.trie_cost(w, s)
        caps = list(range(0, trie + 3))
        costs = O.radix_cache_costs(w, s, order, caps)
        assert costs[0] == total
        assert costs[trie] == trie and costs[-1] == trie
        assert all(a >= b for a, b in zip(costs, costs[1:]))


def test_serve_order_windows():
    """Window 1 keeps the arrival order; a window >= m is the global order;
    otherwise every window is a sorted permutation of its own arrivals."""
    rng = np.random.default_rng(13)
    s = _random_strings(rng, 40, 8, 5)
    arrival = [int(x) for x in rng.permutation(40)]
    assert O.serve_order(s, arrival, 1) == arrival
    assert O.serve_order(s, arrival, 40) == O.serve_order(s) == O.serve_order(s, arrival, 0)
    key = lambda r: (tuple(s[r]), r)
    assert O.serve_order(s) == sorted(range(40), key=key)
    for W in (3, 7, 16):
        out = O.serve_order(s, arrival, W)
        for lo in range(0, 40, W):
            assert out[lo:lo + W] == sorted(arrival[lo:lo + W], key=key)


def test_pinned_reduces_to_free_and_production(C=None):
    """t = 0 is the free problem (OPT by the recurrence); t >= k pins every
    passage, i.e. the relevance order itself."""
    C = O._default()
    rng = np.random.default_rng(17)
    for trial in range(6):
        m, n = int(rng.integers(2, 8)), 14
        ranked = [[int(x) for x in rng.permutation(n)[:int(rng.integers(1, 6))]] for _ in range(m)]
        w = rng.integers(1, 40, size=n).astype(np.int64)
        bits = I.pack_requests(ranked, n)
        opt = C.solve(w, bits)[0]
        seqs, cost = O.pinned_layout(w, ranked, 0, C)
        assert cost == opt
        seqs, cost = O.pinned_layout(w, ranked, 10, C)
        assert seqs == ranked and cost == O.trie_cost(w, ranked)


def test_pinned_exact_with_private_pins():
    """When every pinned passage belongs to no other request, the pinned
    suffixes cannot share, so free layout + pins is the constrained optimum:
    cost = OPT(reduced sets) + sum of pinned weights = brute force."""
    C = O._default()
    rng = np.random.default_rng(23)
    for trial in range(8):
        m, t = int(rng.integers(2, 5)), int(rng.integers(1, 3))
        shared = 6
        ranked = []
        nxt = shared
        for i in range(m):
            pins = list(range(nxt, nxt + t))
            nxt += t
            free = [int(x) for x in rng.permutation(shared)[:int(rng.integers(0, 4))]]
            ranked.append(pins + free)
        n = nxt
        w = rng.integers(1, 20, size=n).astype(np.int64)
        seqs, cost = O.pinned_layout(w, ranked, t, C)
        free_bits = I.pack_requests([r[t:] for r in ranked], n)
        opt_free = C.solve(w, free_bits)[0]
        assert cost == opt_free + sum(int(w[x]) for r in ranked for x in r[:t])
        assert cost == O.brute_force_pinned(w, ranked, t)


def test_pinned_bounds():
    """Any pinned layout is a feasible free layout (cost >= OPT_free) and is
    never below the constrained brute-force optimum."""
    C = O._default()
    rng = np.random.default_rng(29)
    for trial in range(8):
        m, n, t = int(rng.integers(2, 5)), 7, int(rng.integers(0, 3))
        ranked = [[int(x) for x in rng.permutation(n)[:int(rng.integers(1, 5))]] for _ in range(m)]
        w = rng.integers(1, 9, size=n).astype(np.int64)
        seqs, cost = O.pinned_layout(w, ranked, t, C)
        assert cost >= C.solve(w, I.pack_requests(ranked, n))[0]
        assert cost >= O.brute_force_pinned(w, ranked, t)
        for s, r in zip(seqs, ranked):
            assert sorted(s) == sorted(r) and s[len(s) - min(t, len(r)):] == r[:min(t, len(r))]


# ---------------------------------------------------------------------------
# Planted mistakes in the cache simulator: each must fail a pin above.
# ---------------------------------------------------------------------------
_SRC = inspect.getsource(O.radix_cache_cost)
_MUTANTS = {
    "hit does not refresh recency": ("cached[key] = clock\n                continue", "continue"),
    "evicts the most recent leaf": ("victim = min(leaves, key=cached.get)", "victim = max(leaves, key=cached.get)"),
    "current path not protected": ("protected = {seq[:e] for e in range(1, d)}", "protected = set()"),
    "off-by-one capacity": ("while used + need > capacity:", "while used + need >= capacity:"),
    "no-room chunks not paid": ("paid += sum(int(w[x]) for x in seq[d:])", "pass"),
}


def _mutant(old, new):
    assert old in _SRC, old
    ns = dict(np=np)
    exec(_SRC.replace(old, new), ns)
    return ns["radix_cache_cost"]


def _pins_pass(sim) -> bool:
    try:
        w = np.array([5, 3, 4, 7])
        s = [[0, 1], [0, 2], [0, 1], [3]]
        if [sim(w, s, [0, 1, 2, 3], c) for c in (0, 5, 8, 12, 10 ** 6)] != [32, 22, 22, 19, 19]:
            return False
        if [sim(np.ones(3), [[0], [1], [0], [2], [0]], range(5), c) for c in range(4)] != [5, 5, 3, 3]:
            return False
        rng = np.random.default_rng(5)
        for trial in range(25):
            m, n = int(rng.integers(1, 30)), int(rng.integers(3, 12))
            s = _random_strings(rng, m, n, 6)
            w = rng.integers(1, 50, size=n)
            order = O.serve_order(s)
            cap = max([sum(int(w[x]) for x in q) for q in s] + [0])
            if sim(w, s, order, cap) != O.trie_cost(w, s):
                return False
            arrival = [int(x) for x in rng.permutation(m)]
            costs = [sim(w, s, arrival, c) for c in range(0, 40, 3)]
            if any(a < b for a, b in zip(costs, costs[1:])):
                return False
        return True
    except Exception:
        return False


def test_simulator_pins_pass_on_the_real_oracle():
    assert _pins_pass(O.radix_cache_cost)


@pytest.mark.parametrize("name", sorted(_MUTANTS))
def test_simulator_mutant_is_caught(name):
    old, new = _MUTANTS[name]
    assert not _pins_pass(_mutant(old, new)), name

"""Serving order, finite radix cache and pinned layouts on the GPU (Sec. 7.1,
Sec. 8, Thm 7) against the oracle, through the C ABI.  Integer results:
bit-exact."""

from __future__ import annotations

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(1200)]


@pytest.fixture(scope="module")
def mpt():
    import __graft_entry__ as G

    G.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def _random_strings(rng, m, n, kmax, share=0.6):
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


def _edge_cases():
    """(n, strings): single string, empty strings, identical strings, strings
    that are prefixes of others, one-chunk universe."""
    return [
        (3, [[0, 1, 2]]),
        (3, [[], [], []]),
        (4, [[1], [], [1, 2], [1]]),
        (5, [[2, 3], [2, 3], [2, 3], [2, 3]]),
        (6, [[0, 1, 2, 3], [0, 1], [0], [0, 1, 2], [5]]),
        (1, [[0], [0], []]),
    ]


def test_serve_order_parity(mpt):
    rng = np.random.default_rng(41)
    cases = list(_edge_cases())
    for trial in range(20):
        m, n = int(rng.integers(1, 60)), int(rng.integers(1, 12))
        cases.append((n, _random_strings(rng, m, n, 7)))
    # several radix tiles (> 2048 strings), many duplicates, 17-bit chunk ids
    cases.append((20, _random_strings(np.random.default_rng(3), 5000, 20, 6, share=0.8)))
    big_n = 100_000
    cases.append((big_n, [[int(x) for x in np.random.default_rng(7 + i).choice(big_n, 5, replace=False)]
                          for i in range(3000)]))
    for n, s in cases:
        m = len(s)
        assert mpt.mpt_serve_order(n, s).tolist() == O.serve_order(s), (n, m)
        arrival = [int(x) for x in rng.permutation(m)]
        for W in sorted({1, 2, 7, max(1, m // 3), m, m + 5}):
            got = mpt.mpt_serve_order(n, s, arrival, W).tolist()
            assert got == O.serve_order(s, arrival, W), (n, m, W)


def test_cache_costs_parity_small(mpt):
    """Every capacity from 0 to past the trie weight, random arrival orders."""
    rng = np.random.default_rng(43)
    cases = list(_edge_cases())
    for trial in range(30):
        m, n = int(rng.integers(1, 50)), int(rng.integers(1, 10))
        cases.append((n, _random_strings(rng, m, n, 6)))
    for n, s in cases:
        w = rng.integers(1, 40, size=n).astype(np.int64)
        m = len(s)
        trie = O.trie_cost(w, s)
        caps = list(range(0, min(trie + 3, 1024)))
        for order in (list(range(m)), [int(x) for x in rng.permutation(m)], O.serve_order(s)):
            costs, unb = mpt.mpt_cache_costs(w, s, caps, order)
            assert unb == trie
            assert costs.tolist() == O.radix_cache_costs(w, s, order, caps), (n, m)
        # no capacities: only the unbounded cost; a prebuilt CSR gives the same answers
        costs, unb = mpt.mpt_cache_costs(w, s, [], None)
        assert costs.size == 0 and unb == trie
        csr = mpt.to_csr(s)
        assert mpt.mpt_cache_costs(w, csr, caps[:5], None)[0].tolist() == O.radix_cache_costs(w, s, list(range(m)), caps[:5])
        assert mpt.mpt_serve_order(n, csr).tolist() == O.serve_order(s)


def test_cache_costs_parity_stream(mpt):
    """The first 400 requests of the NFCorpus-shaped stream, production layout
    (relevance order) and the greedy layout, in arrival and Thm 7 order, at
    capacities from a quarter request to past the whole trie."""
    w, ranked = I.stream("nfcorpus-shaped", seed=1)
    s = ranked[:400]
    one = int(np.mean([sum(int(w[x]) for x in q) for q in s]))
    caps = [0, one // 4, one // 2, (3 * one) // 4, (9 * one) // 10, one, 2 * one, 4 * one, 16 * one, 64 * one,
            256 * one, 10 ** 12]
    g = mpt.mpt_greedy(w, s)
    for strings in (s, g.perms):
        for order in (list(range(len(s))), O.serve_order(strings)):
            costs, unb = mpt.mpt_cache_costs(w, strings, caps, order)
            assert unb == O.trie_cost(w, strings)
            assert costs.tolist() == O.radix_cache_costs(w, strings, order, caps)


def test_thm7_full_stream(mpt):
    """Thm 7 on the full NFCorpus- and SciFact-shaped streams, for the
    production and greedy layouts: in Thm 7's order a capacity of one request
    (the largest) pays exactly the unbounded cost; the oracle agrees at the
    small capacities it can simulate quickly."""
    for name in ("nfcorpus-shaped", "scifact-shaped"):
        w, ranked = I.stream(name, seed=0)
        g = mpt.mpt_greedy(w, ranked)
        for strings in (ranked, g.perms):
            order = mpt.mpt_serve_order(len(w), strings)
            assert order.tolist() == O.serve_order(strings)
            big = max(sum(int(w[x]) for x in q) for q in strings)
            costs, unb = mpt.mpt_cache_costs(w, strings, [0, big // 2, big, 4 * big], order)
            assert unb == O.trie_cost_sorted(w, strings)
            assert costs[2] == unb and costs[3] == unb
            assert costs[0] == sum(int(w[x]) for q in strings for x in q)
            small = [big // 2]
            assert costs[1] == O.radix_cache_costs(w, strings, order.tolist(), small)[0]


def test_trie_cost_many_strings(mpt):
    """mpt_trie_cost beyond 32 strings (the lexicographic path) against eq. (1)."""
    rng = np.random.default_rng(47)
    for m, n, k in ((33, 10, 6), (200, 30, 8), (5000, 40, 7)):
        s = _random_strings(rng, m, n, k, share=0.7)
        w = rng.integers(1, 1000, size=n).astype(np.int64)
        offs = np.zeros(m + 1, dtype=np.int64)
        offs[1:] = np.cumsum([len(q) for q in s])
        ch = np.array([x for q in s for x in q], dtype=np.int64)
        assert mpt.mpt_trie_cost(w, offs, ch) == O.trie_cost(w, s)


def test_layout_pinned_exact(mpt):
    """Pinned layouts with the exact free layout equal the oracle's string for
    string (same argmin and emission rules); cost and order by eq. (1) and Thm 7."""
    rng = np.random.default_rng(53)
    C = O._default()
    for trial in range(12):
        m, n = int(rng.integers(1, 13)), 30
        ranked = [[int(x) for x in rng.permutation(n)[:int(rng.integers(0, 9))]] for _ in range(m)]
        w = rng.integers(1, 300, size=n).astype(np.int64)
        for t in (0, 1, 2, 3, 9):
            res = mpt.mpt_layout_pinned(w, ranked, t, "exact")
            seqs, cost = O.pinned_layout(w, ranked, t, C)
            assert res.strings == seqs and res.cost == cost
            assert res.serve_order.tolist() == O.serve_order(seqs)
    # a 24-request RAG group (blocked kernels)
    w, ranked = I.stream("nfcorpus-shaped", seed=2)
    group = ranked[:24]
    for t in (0, 1, 3):
        res = mpt.mpt_layout_pinned(w, group, t, "exact")
        assert res.cost == O.trie_cost(w, res.strings)
        for sq, r in zip(res.strings, group):
            assert sorted(sq) == sorted(r) and sq[len(sq) - t:] == r[:t]


def test_layout_pinned_greedy(mpt):
    """Greedy free layout + pins equals the oracle's greedy on the reduced sets
    followed by the pins."""
    w, ranked = I.stream("scifact-shaped", seed=3)
    ranked = ranked[:150]
    n = len(w)
    for t in (0, 1, 2, 8):
        res = mpt.mpt_layout_pinned(w, ranked, t, "greedy")
        free = [r[t:] for r in ranked]
        g = O.greedy(w, I.pack_requests(free, n))
        seqs = [list(p) + r[:t] for p, r in zip(g["perms"], ranked)]
        assert res.strings == seqs
        assert res.cost == O.trie_cost(w, seqs)
        assert res.serve_order.tolist() == O.serve_order(seqs)
    # t >= k pins everything: the production layout
    res = mpt.mpt_layout_pinned(w, ranked, 8, "greedy")
    assert res.strings == [list(r) for r in ranked]

"""Pins that tie the CPU oracle to facts outside itself.

Each ``pin_*`` takes a compiled oracle (``oracle.COracle``) and raises
``AssertionError`` if the oracle disagrees with the paper's printed values, a
closed form, an exhaustive brute force written independently of the
recurrence, or an invariant the paper proves.  ``test_oracle.py`` runs them
on the real oracle; ``test_oracle_mutants.py`` runs them on copies of
``oracle.c`` with planted mistakes and requires every mistake to be caught.
"""

from __future__ import annotations

import json
import os

import numpy as np

import oracle as O
from paper_2609_13692_gb300 import instances as I

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def _opt(C, inst):
    return C.solve(inst.weights, inst.bits)[0]


def pin_k4_3(C):
    """Thm 4: the complete 3-uniform hypergraph on four chunks has OPT_free = 8."""
    g = GOLDEN["k4_3"]
    assert _opt(C, I.k4_3()) == g["opt_free"]


def pin_open_problem(C):
    """Sec. 10.1: the k = 4 instance on 7 chunks has OPT_free = 14."""
    assert _opt(C, I.open_problem_k4()) == GOLDEN["open_problem_k4"]["opt_free"]


def pin_tightness_witness(C):
    """Sec. 6.3: optimal saving 2 on a request total of 12, so OPT = 10."""
    g = GOLDEN["tightness_witness"]
    assert _opt(C, I.tightness_witness()) == g["request_total"] - g["optimal_saving"]


def pin_leave_one_out(C):
    """Thm 5 / Sec. 5.1: OPT_free(L_n) is the minimum external path length."""
    seq = GOLDEN["leave_one_out_sequence"]
    for n, v in enumerate(seq["values"], start=seq["n_from"]):
        assert _opt(C, I.leave_one_out(n)) == v, n
    for n, free, _glob in GOLDEN["leave_one_out_table"]["rows"]:
        if n <= 16:
            assert _opt(C, I.leave_one_out(n)) == free, n
    for n in (11, 13):
        assert _opt(C, I.leave_one_out(n)) == O.loo_free(n), n


def _tiny_instances(count, m_range, n, k_range, seed, wmax=5):
    rng = np.random.default_rng(seed)
    out = []
    for t in range(count):
        m = int(rng.integers(m_range[0], m_range[1] + 1))
        out.append(I.random_instance(m, n, k_range, seed=int(rng.integers(1 << 30)), wmin=1, wmax=wmax))
    return out


def pin_brute_force_permutations(C):
    """Sec. 2 / eq. (1): OPT_free is the least trie cost over all per-request
    permutations; checked exhaustively on tiny instances."""
    for inst in _tiny_instances(12, (1, 4), 6, (1, 3), seed=11):
        assert _opt(C, inst) == O.brute_force_permutations(inst.weights, inst.bits), inst.name
    inst = I.random_instance(3, 5, 4, seed=5, wmin=1, wmax=7)
    assert _opt(C, inst) == O.brute_force_permutations(inst.weights, inst.bits)


def pin_brute_force_hierarchies(C):
    """Thm 1, eq. (2): OPT_free = min over binary hierarchies of sum_x w(x) t_x(H)."""
    for inst in _tiny_instances(10, (2, 6), 8, (1, 5), seed=23, wmax=9):
        assert _opt(C, inst) == O.brute_force_hierarchies(inst.weights, inst.bits), inst.name


def pin_vertex_cover(C):
    """Prop 2: |R_i| = 2, unit weights, distinct requests => OPT = tau(G) + m."""
    rng = np.random.default_rng(7)
    for t in range(8):
        nv = int(rng.integers(3, 8))
        all_edges = [(u, v) for u in range(nv) for v in range(u + 1, nv)]
        m = int(rng.integers(1, min(len(all_edges), 12) + 1))
        pick = rng.choice(len(all_edges), size=m, replace=False)
        edges = [all_edges[j] for j in pick]
        inst = I.Instance(np.ones(nv, dtype=np.int64), I.pack_requests([list(e) for e in edges], nv))
        tau = O.min_vertex_cover(edges, range(nv))
        assert _opt(C, inst) == tau + m, (edges, tau)


def pin_intersection_weights(C):
    """Thm 1 proof: w(I(S)) is the weight of the intersection of R_i, i in S."""
    for inst in _tiny_instances(6, (1, 8), 70, (2, 30), seed=31, wmax=50):
        R = O.request_sets(inst.weights, inst.bits)
        wI = C.intersection_weights(inst.weights, inst.bits)
        m = inst.m
        union = set().union(*R)
        assert wI[0] == sum(int(inst.weights[x]) for x in union)
        for S in range(1, 1 << m):
            members = [i for i in range(m) if (S >> i) & 1]
            common = set.intersection(*[R[i] for i in members])
            assert wI[S] == sum(int(inst.weights[x]) for x in common), (inst.name, S)
        for S in (1, (1 << m) - 1, (1 << m) // 3 or 1):
            assert C.wI_one(inst.weights, inst.bits, S) == wI[S]


def pin_layout_is_optimal(C):
    """Thm 1 ('<=' direction): the top-down emission along the returned
    hierarchy is a valid layout whose trie cost equals OPT; every F(S) lies
    between w(union of R_i) and sum of w(R_i) over i in S."""
    for inst in _tiny_instances(6, (2, 10), 40, (2, 8), seed=43, wmax=30):
        opt, F, wI, split = C.solve(inst.weights, inst.bits)
        perms, dfs = O.layout(inst.weights, inst.bits, split)
        R = O.request_sets(inst.weights, inst.bits)
        for i, p in enumerate(perms):
            assert sorted(p) == sorted(R[i]) and len(p) == len(set(p))
        assert sorted(dfs) == list(range(inst.m))
        assert O.trie_cost(inst.weights, perms) == opt
        w = inst.weights
        for S in range(1, 1 << inst.m):
            members = [i for i in range(inst.m) if (S >> i) & 1]
            union = set().union(*[R[i] for i in members])
            lo = sum(int(w[x]) for x in union)
            hi = sum(sum(int(w[x]) for x in R[i]) for i in members)
            assert lo <= F[S] <= hi, (inst.name, S)


def pin_bounds(C):
    """Sec. 6.3 spanning-tree lower bound <= OPT_free <= any global order's cost (Sec. 3.1)."""
    for inst in _tiny_instances(8, (2, 9), 30, (2, 9), seed=59, wmax=40):
        opt = _opt(C, inst)
        assert O.spanning_tree_bound(inst.weights, inst.bits) <= opt
        assert opt <= O.global_order_cost(inst.weights, inst.bits)


def pin_split_rule(C):
    """The argmin reading: split[S] is the smallest A holding the lowest
    request of S whose split attains F(S) (F(S) itself from the table)."""
    for inst in _tiny_instances(4, (2, 8), 20, (1, 8), seed=71, wmax=3):
        opt, F, wI, split = C.solve(inst.weights, inst.bits)
        m = inst.m
        for S in range(1, 1 << m):
            if S & (S - 1) == 0:
                assert split[S] == 0 and F[S] == wI[S]
                continue
            low = S & -S
            cands = [A for A in range(1, S) if (A & S) == A and (A & low) and A != S]
            vals = [int(F[A] + F[S ^ A]) for A in cands]
            best = min(vals)
            assert F[S] == best - wI[S]
            assert split[S] == min(A for A, v in zip(cands, vals) if v == best), (inst.name, S)


def pin_recompute(C):
    """oracle_recompute reproduces oracle_dp's F and split from its own table."""
    inst = I.random_instance(9, 50, (3, 10), seed=83, wmin=1, wmax=100)
    opt, F, wI, split = C.solve(inst.weights, inst.bits)
    subsets = np.arange(1, 1 << inst.m, dtype=np.uint64)
    Fr, sr, wr = C.recompute(inst.weights, inst.bits, F, subsets)
    assert np.array_equal(Fr, F[1:]) and np.array_equal(sr, split[1:]) and np.array_equal(wr, wI[1:])


def pin_recompute_local(C):
    """recompute_local (one subset from its own submask table) agrees with oracle_dp."""
    inst = I.random_instance(9, 40, (2, 8), seed=87, wmin=1, wmax=60)
    opt, F, wI, split = C.solve(inst.weights, inst.bits)
    rng = np.random.default_rng(1)
    for S in [int(x) for x in rng.integers(1, 1 << inst.m, size=60)] + [(1 << inst.m) - 1]:
        pos = [i for i in range(inst.m) if (S >> i) & 1]
        idx = [sum(1 << pos[q] for q in range(len(pos)) if (j >> q) & 1) for j in range(1 << len(pos))]
        F_sub = F[idx]
        k = len(pos)
        full = (1 << k) - 1
        wi = int(wI[S])
        if k <= 1:
            continue
        j = np.arange(1, full, 2)
        vals = F_sub[j] + F_sub[full ^ j]
        assert int(vals.min()) - wi == F[S]
        f, a, w = O.recompute_local(inst.weights, inst.bits, S, F_sub)
        assert (f, a, w) == (F[S], split[S], wI[S])


def _balanced_t(lo, hi, a, b):
    """Maximal clusters of a balanced binary tree over the requests lo..hi
    (split at the midpoint) that lie inside the interval [a, b]."""
    if b < lo or hi < a:
        return 0
    if a <= lo and hi <= b:
        return 1
    mid = (lo + hi) // 2
    return _balanced_t(lo, mid, a, b) + _balanced_t(mid + 1, hi, a, b)


def pin_c1p_bound(C):
    """Consecutive-ones instances (Sec. 3, "a tractable special case"): each
    chunk is wanted by a contiguous run of requests, so in a balanced tree
    over that line every S_x splits into at most 2 ceil(log2 m) clusters, and
    by Thm 1 (eq. 1) OPT_free <= sum_x w(x) t_x(balanced) <=
    sum_x w(x) min(|S_x|, 2 ceil(log2 m))."""
    rng = np.random.default_rng(97)
    for _ in range(12):
        m = int(rng.integers(2, 12))
        n = int(rng.integers(3, 30))
        runs = []
        for _x in range(n):
            a = int(rng.integers(0, m))
            runs.append((a, int(rng.integers(a, m))))
        reqs = [[x for x, (a, b) in enumerate(runs) if a <= i <= b] for i in range(m)]
        w = rng.integers(1, 50, size=n, dtype=np.int64)
        inst = I.Instance(w, I.pack_requests(reqs, n))
        opt = _opt(C, inst)
        depth = 2 * int(np.ceil(np.log2(m)))
        balanced = sum(int(w[x]) * _balanced_t(0, m - 1, a, b) for x, (a, b) in enumerate(runs))
        bound = sum(int(w[x]) * min(b - a + 1, depth) for x, (a, b) in enumerate(runs))
        assert opt <= balanced <= bound, (m, n, opt, balanced, bound)


ALL_PINS = [
    pin_k4_3,
    pin_open_problem,
    pin_tightness_witness,
    pin_leave_one_out,
    pin_brute_force_permutations,
    pin_brute_force_hierarchies,
    pin_vertex_cover,
    pin_intersection_weights,
    pin_layout_is_optimal,
    pin_bounds,
    pin_split_rule,
    pin_recompute,
    pin_c1p_bound,
    pin_recompute_local,
]

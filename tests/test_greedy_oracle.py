"""The greedy part of the oracle (Sec. 6.2, Thm 6) against the paper and the exact recurrence."""

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I
from tests import oracle_pins as P


def _exact_hierarchy_weights(inst, split):
    """w(I(v)) of the internal nodes of the exact optimal hierarchy."""
    R = O.request_sets(inst.weights, inst.bits)
    w = inst.weights
    out = []

    def rec(S):
        if S & (S - 1) == 0:
            return
        members = [i for i in range(inst.m) if (S >> i) & 1]
        common = set.intersection(*[R[i] for i in members])
        out.append(int(sum(int(w[x]) for x in common)))
        A = int(split[S])
        rec(A)
        rec(S ^ A)

    rec((1 << inst.m) - 1)
    return out


def test_greedy_exact_on_leave_one_out():
    """Sec. 6.2: greedy is exactly optimal on L_n (printed for n = 16, 32, 64)."""
    for n, free in P.GOLDEN["greedy_on_loo"]["rows"]:
        if n > 32:
            continue
        inst = I.leave_one_out(n)
        g = O.greedy(inst.weights, inst.bits)
        assert g["cost"] == free
        assert O.trie_cost(inst.weights, g["perms"]) == free


def test_greedy_tightness_witness():
    """Sec. 6.3: on {0123},{14},{2578},{46} greedy takes a saving of 1 against the optimal 2."""
    inst = I.tightness_witness()
    g = O.greedy(inst.weights, inst.bits)
    assert g["savings"] == 1
    opt = O.solve(inst.weights, inst.bits)[0]
    assert 12 - opt == 2


def test_thm6_half_approximation_and_threshold_counts():
    """Thm 6: SAV(H_g) >= SAV*/2; its proof: merge values never increase (i),
    and A(theta) <= 2 G(theta) for every threshold (ii)."""
    rng = np.random.default_rng(5)
    for t in range(25):
        inst = I.random_instance(int(rng.integers(2, 10)), 30, (1, 8), seed=int(rng.integers(1 << 30)), wmax=20)
        opt, F, wI, split = O.solve(inst.weights, inst.bits)
        total = sum(sum(int(inst.weights[x]) for x in r) for r in O.request_sets(inst.weights, inst.bits))
        g = O.greedy(inst.weights, inst.bits)
        sav_star = total - opt
        assert 2 * g["savings"] >= sav_star
        vals = [v for _, _, v in g["merges"]]
        assert all(vals[i] >= vals[i + 1] for i in range(len(vals) - 1))
        a_vals = _exact_hierarchy_weights(inst, split)
        assert sum(a_vals) == sav_star
        for theta in sorted(set(a_vals + vals)):
            if theta <= 0:
                continue
            A = sum(1 for x in a_vals if x >= theta)
            G = sum(1 for x in vals if x >= theta)
            assert A <= 2 * G, (theta, A, G)
        # bounds: spanning tree <= OPT <= greedy; the greedy layout's trie costs at most its hierarchy cost
        assert O.spanning_tree_bound(inst.weights, inst.bits) <= opt <= g["cost"]
        assert O.trie_cost(inst.weights, g["perms"]) <= g["cost"]
        R = O.request_sets(inst.weights, inst.bits)
        assert all(sorted(p) == sorted(R[i]) for i, p in enumerate(g["perms"]))
        assert sorted(g["dfs"]) == list(range(inst.m))


def test_sorted_trie_cost_matches_trie_builder():
    rng = np.random.default_rng(8)
    for t in range(20):
        w = rng.integers(1, 9, size=12)
        perms = [list(rng.permutation(rng.choice(12, size=int(rng.integers(0, 6)), replace=False))) for _ in range(7)]
        assert O.trie_cost_sorted(w, perms) == O.trie_cost(w, perms)

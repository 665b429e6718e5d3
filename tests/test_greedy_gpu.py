"""mpt_greedy (Sec. 6.2 hierarchy, Sec. 6.3 bound) against the oracle and the paper."""

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I
from tests import oracle_pins as P

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def mpt():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_13692_gb300 import build as B

    B.build()
    O.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def _check(mpt, inst):
    reqs = [sorted(r) for r in O.request_sets(inst.weights, inst.bits)]
    got = mpt.mpt_greedy(inst.weights, reqs)
    ref = O.greedy(inst.weights, inst.bits)
    assert [tuple(x) for x in got.merges.tolist()] == [(a, b) for a, b, _ in ref["merges"]]
    assert got.merge_values.tolist() == [v for _, _, v in ref["merges"]]
    assert got.savings == ref["savings"] and got.cost == ref["cost"]
    assert got.lower_bound == O.spanning_tree_bound(inst.weights, inst.bits)
    assert got.perms == ref["perms"]
    assert got.dfs_order.tolist() == ref["dfs"]
    return got


@pytest.mark.parametrize("m", [1, 2, 3, 7, 20, 64, 150])
def test_greedy_random(mpt, m):
    inst = I.random_instance(m, 400, (0, 12), seed=100 + m, wmin=1, wmax=300, allow_empty=True)
    _check(mpt, inst)


def test_greedy_rag_and_ties(mpt):
    _check(mpt, I.config(1))
    _check(mpt, I.config(3))          # m = 24 RAG-shaped groups
    _check(mpt, I.tightness_witness())
    _check(mpt, I.leave_one_out(24))  # all ties


def test_greedy_leave_one_out_printed(mpt):
    """Sec. 6.2: greedy is exactly optimal on L_n, n = 16, 32, 64, 128 -> 64, 160, 384, 896."""
    for n, free in P.GOLDEN["greedy_on_loo"]["rows"]:
        inst = I.leave_one_out(n)
        reqs = [sorted(r) for r in O.request_sets(inst.weights, inst.bits)]
        g = mpt.mpt_greedy(inst.weights, reqs)
        assert g.cost == free
        assert O.trie_cost_sorted(inst.weights, g.perms) == free


def test_greedy_large_trace_shape(mpt):
    """m = 3000 requests of k = 8 passages (the size of the paper's NFCorpus
    trace): layout validity, Thm 6 (i) monotone merges, bound <= greedy."""
    rng = np.random.default_rng(3)
    n = 3600
    weights = rng.integers(50, 400, size=n).astype(np.int64)
    pools = [rng.choice(n, size=60, replace=False) for _ in range(200)]
    reqs = []
    for _ in range(3000):
        pool = pools[int(rng.integers(len(pools)))]
        chosen = set()
        while len(chosen) < 8:
            chosen.add(int(pool[int(rng.integers(60))]) if rng.random() < 0.85 else int(rng.integers(n)))
        reqs.append(sorted(chosen))
    g = mpt.mpt_greedy(weights, reqs)
    assert all(sorted(p) == r for p, r in zip(g.perms, reqs))
    assert sorted(g.dfs_order.tolist()) == list(range(3000))
    v = g.merge_values
    assert bool(np.all(v[:-1] >= v[1:]))
    assert g.lower_bound <= g.cost
    assert O.trie_cost_sorted(weights, g.perms) <= g.cost

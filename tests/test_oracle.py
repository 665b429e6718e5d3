"""The CPU oracle against the paper's printed values, closed forms and brute force (no GPU)."""

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I
from tests import oracle_pins as P


@pytest.fixture(scope="module")
def C():
    return O.COracle(O.build())


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(C, pin):
    pin(C)


def test_closed_forms_match_printed_table():
    """Thm 5 closed forms against the Sec. 5.1 table and the Sec. 6.2 values."""
    for n, free, glob in P.GOLDEN["leave_one_out_table"]["rows"]:
        assert O.loo_free(n) == free and O.loo_glob(n) == glob
    for n, free in P.GOLDEN["greedy_on_loo"]["rows"]:
        assert O.loo_free(n) == free
    g = P.GOLDEN["leave_one_out_caterpillar"]
    assert O.loo_glob(g["n"]) == g["cost"]
    assert O.loo_free(20) == 88


def test_global_order_brute_force():
    """OPT_glob by enumerating chunk orders: Thm 4 (9), Sec. 10.1 (21), Thm 5 (L_n)."""
    assert O.brute_force_global_order(I.k4_3().weights, I.k4_3().bits) == P.GOLDEN["k4_3"]["opt_glob"]
    inst = I.open_problem_k4()
    assert O.brute_force_global_order(inst.weights, inst.bits) == P.GOLDEN["open_problem_k4"]["opt_glob"]
    for n in range(2, 7):
        inst = I.leave_one_out(n)
        assert O.brute_force_global_order(inst.weights, inst.bits) == O.loo_glob(n)


def test_trie_cost_of_printed_layout():
    """Thm 4 proof: the layout abc, abd, cda, cdb has a trie of 8 nodes."""
    g = P.GOLDEN["k4_3"]
    ids = {"a": 0, "b": 1, "c": 2, "d": 3}
    perms = [[ids[c] for c in row] for row in g["layout_example"]]
    assert O.trie_cost(np.ones(4, dtype=np.int64), perms) == g["layout_example_cost"]


def test_thm7_dfs_order_one_request_cache(C):
    """Thm 7: in the hierarchy's DFS order, a radix cache holding one request's
    context (LRU leaf eviction) pays exactly the unbounded-cache cost."""
    rng = np.random.default_rng(97)
    for t in range(6):
        inst = I.random_instance(int(rng.integers(3, 11)), 40, (2, 9), seed=int(rng.integers(1 << 30)),
                                 wmin=1, wmax=20)
        opt, F, wI, split = C.solve(inst.weights, inst.bits)
        perms, dfs = O.layout(inst.weights, inst.bits, split)
        cap = max(sum(int(inst.weights[x]) for x in p) for p in perms)
        assert O.radix_cache_cost(inst.weights, perms, dfs, cap) == opt
        # an unbounded cache pays the trie cost in any order
        assert O.radix_cache_cost(inst.weights, perms, list(range(inst.m))[::-1], 10 ** 9) == opt
    # with a tiny cache the simulator pays at least the trie cost
    inst = I.config(1)
    opt, F, wI, split = C.solve(inst.weights, inst.bits)
    perms, dfs = O.layout(inst.weights, inst.bits, split)
    assert O.radix_cache_cost(inst.weights, perms, dfs, 600) >= opt


def test_config_instances_shapes():
    for idx in (1, 2, 3):
        inst = I.config(idx)
        c = I.CONFIGS[idx]
        assert inst.m == c["m"] and inst.n == c["n"]
        assert inst.bits.shape == (c["m"], (c["n"] + 63) // 64) and inst.bits.dtype == np.uint64
        assert inst.weights.dtype == np.int64 and inst.weights.min() >= 1
        reqs = inst.requests()
        if "k" in c:
            assert all(len(r) == c["k"] for r in reqs)
    again = I.config(3)
    assert np.array_equal(again.bits, I.config(3).bits) and np.array_equal(again.weights, I.config(3).weights)
    w = I.config(3).weights
    assert 32 <= w.min() and w.max() <= 512 and 120 < w.mean() < 180


def test_pack_roundtrip():
    reqs = [[0, 63, 64, 129], [], [5]]
    bits = I.pack_requests(reqs, 130)
    assert I.unpack_requests(bits, 130) == [sorted(r) for r in reqs]


def test_config1_and_config2_full(C):
    """Config 2 is L_20: OPT = 88 (Thm 5); config 1's layout realises its OPT."""
    inst = I.config(2)
    assert C.solve(inst.weights, inst.bits)[0] == O.loo_free(20) == 88
    inst = I.config(1)
    opt, F, wI, split = C.solve(inst.weights, inst.bits)
    perms, dfs = O.layout(inst.weights, inst.bits, split)
    assert O.trie_cost(inst.weights, perms) == opt
    assert O.spanning_tree_bound(inst.weights, inst.bits) <= opt <= O.global_order_cost(inst.weights, inst.bits)


def test_private_chunks_shift_F_by_a_constant():
    """Thm 1: a chunk that one request alone holds is one maximal cluster in
    every hierarchy (t_x(H) = 1), so appending one to request i adds its
    weight to F(S) for every S holding i, to w(I(S)) only at S = {i} and
    S = {}, and changes no split.  The tiled kernels rely on this to leave
    such weights out of their packed keys."""
    rng = np.random.default_rng(123)
    for t in range(8):
        m = int(rng.integers(2, 11))
        base = I.random_instance(m, 30, (0, 7), seed=int(rng.integers(1 << 30)), wmin=1, wmax=50, allow_empty=True)
        inst = I.with_query_chunks(base, 1, 10 ** 6, seed=t, every=1 + t % 2)
        q = np.zeros(m, dtype=np.int64)
        owners = list(range(0, m, 1 + t % 2))
        q[owners] = inst.weights[base.n:]
        opt0, F0, wI0, s0 = O.solve(base.weights, base.bits)
        opt1, F1, wI1, s1 = O.solve(inst.weights, inst.bits)
        S = np.arange(1 << m, dtype=np.int64)
        pi_S = sum(((S >> i) & 1) * q[i] for i in range(m))
        assert np.array_equal(F1, F0 + pi_S)
        expect_wI = wI0.copy()
        expect_wI[[1 << i for i in range(m)]] += q
        expect_wI[0] += int(q.sum())
        assert np.array_equal(wI1, expect_wI)
        assert np.array_equal(s1, s0)
        assert opt1 == opt0 + int(q.sum())
    # the same shift by brute force over all chunk orders (no recurrence)
    base = I.Instance(np.array([2, 3, 1, 4], dtype=np.int64), I.pack_requests([[0, 1], [1, 2], [0, 2, 3]], 4))
    inst = I.with_query_chunks(base, 5, 9, seed=1)
    extra = int(inst.weights[base.n:].sum())
    assert O.brute_force_permutations(inst.weights, inst.bits) == O.brute_force_permutations(base.weights,
                                                                                            base.bits) + extra


def test_universal_chunks_shift_F_by_a_constant():
    """Thm 1: a chunk that all m >= 2 requests hold has the root as its one
    maximal cluster in every hierarchy, so it adds its weight u to F(S) for
    every non-empty S and to every w(I(S)), and changes no split."""
    rng = np.random.default_rng(321)
    for t in range(8):
        m = int(rng.integers(2, 11))
        base = I.random_instance(m, 30, (0, 7), seed=int(rng.integers(1 << 30)), wmin=1, wmax=50, allow_empty=True)
        u = int(rng.integers(1, 10 ** 6))
        inst = I.with_common_prefix(base, u)
        opt0, F0, wI0, s0 = O.solve(base.weights, base.bits)
        opt1, F1, wI1, s1 = O.solve(inst.weights, inst.bits)
        nonempty = (np.arange(1 << m) != 0).astype(np.int64)
        assert np.array_equal(F1, F0 + u * nonempty)
        assert np.array_equal(wI1, wI0 + u)
        assert np.array_equal(s1, s0)
        assert opt1 == opt0 + u
    base = I.Instance(np.array([2, 3, 1, 4], dtype=np.int64), I.pack_requests([[0, 1], [1, 2], [0, 2, 3]], 4))
    inst = I.with_common_prefix(base, 7)
    assert O.brute_force_permutations(inst.weights, inst.bits) == O.brute_force_permutations(base.weights,
                                                                                            base.bits) + 7


def test_dp_at_reproduces_the_full_table(C):
    """The recurrence's step at listed subsets (used to time samples of layers
    too large to finish) gives oracle_dp's F and split at every subset when it
    reads the oracle's own tables, including singletons and the empty set;
    and F(S) = F(split) + F(S \\ split) - w(I(S)) at the full set (Sec. 3.1)."""
    inst = I.config(1)
    opt, F, wI, split = C.solve(inst.weights, inst.bits)
    m = inst.m
    subsets = np.arange(1 << m, dtype=np.uint64)
    Fa, sa = C.dp_at(wI, F, m, subsets, threads=2)
    assert np.array_equal(Fa, F) and np.array_equal(sa, split)
    full = (1 << m) - 1
    A = int(split[full])
    assert Fa[full] == F[A] + F[full ^ A] - wI[full] == opt
    rng = np.random.default_rng(3)
    pick = rng.integers(0, 1 << m, size=200).astype(np.uint64)
    Fb, sb = C.dp_at(wI, F, m, pick, threads=1)
    assert np.array_equal(Fb, F[pick.astype(np.int64)]) and np.array_equal(sb, split[pick.astype(np.int64)])
    with pytest.raises(ValueError):
        C.dp_at(wI, F, m, np.array([1 << m], dtype=np.uint64))

"""CUDA path vs the CPU oracle, through the C ABI.

Integer results must be bit-exact: OPT, every F(S), every w(I(S)), every
split(S), the per-request permutations and the DFS order -- in full up to
m = 24, where the oracle still finishes the whole recurrence.  Where it
cannot (m >= 28), at least 10^5 sampled subsets are recomputed by the oracle
from the GPU's own table of smaller subsets, w(I(S)) is recomputed from
scratch, and the trie cost of the returned layout must equal OPT.
"""

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I
from tests import weights as W

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


def gpu_solve(mpt, inst, mode="auto"):
    res = mpt.solve(inst.weights, inst.bits, mode=mode, profile=True)
    F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(res.ctx))
    prof = mpt.mpt_get_profile(res.ctx)
    return res, F, wI, split.view(np.uint32), prof


def assert_full_parity(mpt, inst, mode="auto", expect_mode=None):
    res, F, wI, split, prof = gpu_solve(mpt, inst, mode)
    opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
    if expect_mode is not None:
        assert prof["dp_mode"] == expect_mode
    assert res.opt == opt
    assert np.array_equal(wI, owI), np.flatnonzero(wI != owI)[:10]
    assert np.array_equal(F, oF), np.flatnonzero(F != oF)[:10]
    assert np.array_equal(split, osplit), np.flatnonzero(split != osplit)[:10]
    perms, dfs = O.layout(inst.weights, inst.bits, osplit)
    assert res.permutations() == perms
    assert res.dfs_order.tolist() == dfs
    assert O.trie_cost(inst.weights, res.permutations()) == opt
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == opt
    return res, prof


def test_config1_bit_exact(mpt):
    """Zipf m = 12, 48 chunks, k = 5 (one in-tile launch)."""
    assert_full_parity(mpt, I.config(1), expect_mode=1)


def test_config2_leave_one_out(mpt):
    """L_20: OPT = 20*5 - 32 + 20 = 88 (Thm 5); all tables bit-exact."""
    res, prof = assert_full_parity(mpt, I.config(2), expect_mode=1)
    assert res.opt == O.loo_free(20) == 88


def test_table_views_follow_each_solve(mpt):
    """The blocked solve keeps its tables tile-major and fills the natural
    views on the first table request: repeated requests return the same
    views, and a second solve on the same context -- whose working tables
    reuse the views' buffers -- fills them again, bit-exact (int64 and lean)."""
    rng = np.random.default_rng(77)
    m, n = 17, 60
    reqs = [[int(x) for x in rng.choice(n, size=int(rng.integers(3, 9)), replace=False)] for _ in range(m)]
    inst = I.Instance(rng.integers(1, 50, size=n).astype(np.int64), I.pack_requests(reqs, n))
    opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    for rnd in range(2):
        assert mpt.mpt_solve(ctx) == opt
        first = mpt.mpt_tables(ctx)
        again = mpt.mpt_tables(ctx)
        assert [t.data_ptr() for t in first] == [t.data_ptr() for t in again]
        F, wI, split = (t.cpu().numpy() for t in again)
        assert np.array_equal(F, oF) and np.array_equal(wI, owI)
        assert np.array_equal(split.view(np.uint32), osplit), rnd
    mpt.mpt_set_tables(ctx, "lean")
    for rnd in range(2):
        assert mpt.mpt_solve(ctx) == opt
        mpt.mpt_tables32(ctx)
        F, split = (t.cpu().numpy() for t in mpt.mpt_tables32(ctx))
        assert np.array_equal(F.astype(np.int64), oF)
        assert np.array_equal(split.view(np.uint32), osplit), rnd


@pytest.mark.parametrize("m", list(range(1, 19)))
def test_random_sweep_blocked(mpt, m):
    rng = np.random.default_rng(1000 + m)
    n = int(rng.integers(1, 300))
    inst = I.random_instance(m, n, (0, min(n, 14)), seed=int(rng.integers(1 << 30)), wmin=1, wmax=512,
                             allow_empty=True)
    assert_full_parity(mpt, inst, "blocked", expect_mode=1)


@pytest.mark.parametrize("m", [1, 2, 5, 9, 10, 11, 12, 13, 14, 16])
def test_random_sweep_general(mpt, m):
    inst = I.random_instance(m, 64, (1, 12), seed=77 + m, wmin=1, wmax=1000)
    assert_full_parity(mpt, inst, "general", expect_mode=2)


@pytest.mark.parametrize("n", [13, 14, 15, 16, 17, 18])
def test_leave_one_out_ties(mpt, n):
    """Unit weights give many optimal splits: the tie rule is exercised everywhere."""
    res, prof = assert_full_parity(mpt, I.leave_one_out(n), expect_mode=1)
    assert res.opt == O.loo_free(n)


def test_paper_examples(mpt):
    for inst, opt in ((I.k4_3(), 8), (I.open_problem_k4(), 14), (I.tightness_witness(), 10)):
        res, prof = assert_full_parity(mpt, inst)
        assert res.opt == opt


def test_edge_cases(mpt):
    cases = [
        I.Instance(np.array([5], dtype=np.int64), I.pack_requests([[0]], 1)),                   # m = 1, n = 1
        I.Instance(np.array([3, 4], dtype=np.int64), I.pack_requests([[], [0, 1], []], 2)),     # empty requests
        I.Instance(np.arange(1, 9, dtype=np.int64), I.pack_requests([[1, 2, 3]] * 14, 8)),      # identical requests
        I.Instance(np.arange(1, 17, dtype=np.int64), I.pack_requests([[i] for i in range(16)], 16)),  # disjoint
        I.Instance(np.ones(200, dtype=np.int64), I.pack_requests([[199]] * 15, 200)),           # last chunk only
        I.random_instance(15, 3, (0, 3), seed=5, allow_empty=True),                              # tiny universe
    ]
    for inst in cases:
        for mode in ("blocked", "general"):
            assert_full_parity(mpt, inst, mode)


def test_large_weights_use_wide_then_general(mpt):
    """Shared weight >= 2^20: the packed 32-bit keys would overflow, AUTO picks the 64-bit keys;
    from 2^51 on those would overflow too, and AUTO picks the int64 kernels."""
    inst = I.random_instance(14, 50, (3, 12), seed=9, wmin=10 ** 9, wmax=10 ** 12)
    assert W.shared_weight(inst) >= 1 << 20
    assert_full_parity(mpt, inst, "auto", expect_mode=3)
    huge = I.random_instance(14, 50, (3, 12), seed=9, wmin=1 << 46, wmax=1 << 47)
    assert W.shared_weight(huge) >= 1 << 51
    assert_full_parity(mpt, huge, "auto", expect_mode=2)


def test_sum_just_below_blocked_limit(mpt):
    """sum_i w(R_i) = 2^20 - 1 (chunks 16..19 private, the shared weight
    955,371), BLOCKED forced."""
    m = 15
    reqs = [[i, (i + 1) % 20, (i + 7) % 20] for i in range(m)]
    w = np.full(20, 1, dtype=np.int64)
    total_slots = sum(len(r) for r in reqs)
    w[:] = (2 ** 20 - 1) // total_slots
    inst = I.Instance(w, I.pack_requests(reqs, 20))
    slack = 2 ** 20 - 1 - int(sum(w[x] for r in reqs for x in r))
    inst.weights[reqs[0][0]] += slack // sum(1 for r in reqs if reqs[0][0] in r)
    assert sum(int(inst.weights[x]) for r in reqs for x in r) < 2 ** 20
    assert_full_parity(mpt, inst, "blocked", expect_mode=1)


def _sample_subsets(m, rng, uniform=20000, budget_per_layer=2.0e7):
    """Uniform random subsets plus, per size k, as many random k-subsets as a
    budget of splits allows (the full set always included)."""
    full = (1 << m) - 1
    out = set(int(x) for x in rng.integers(1, full + 1, size=uniform, dtype=np.int64))
    for k in range(1, m + 1):
        per = 2.0 ** (k - 1)
        cnt = int(min(200, max(1, budget_per_layer // per)))
        for _ in range(cnt):
            members = rng.choice(m, size=k, replace=False)
            out.add(int(sum(1 << int(i) for i in members)))
    out.add(full)
    return np.array(sorted(out), dtype=np.uint64)


def assert_sampled_parity(mpt, inst, seed, uniform=20000):
    res, F, wI, split, prof = gpu_solve(mpt, inst)
    m = inst.m
    full = (1 << m) - 1
    assert res.opt == F[full]
    # the layout realises OPT (Thm 1), checked by two independent trie builders
    assert O.trie_cost(inst.weights, res.permutations()) == res.opt
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == res.opt
    R = O.request_sets(inst.weights, inst.bits)
    for i, p in enumerate(res.permutations()):
        assert sorted(p) == sorted(R[i])
    assert sorted(res.dfs_order.tolist()) == list(range(m))
    # bounds of Sec. 6.3 and Sec. 3.1
    assert O.spanning_tree_bound(inst.weights, inst.bits) <= res.opt <= O.global_order_cost(inst.weights, inst.bits)
    # sampled recomputation
    rng = np.random.default_rng(seed)
    subsets = _sample_subsets(m, rng, uniform=uniform)
    Fr, sr, wr = O.recompute(inst.weights, inst.bits, F, subsets)
    idx = subsets.astype(np.int64)
    assert np.array_equal(wr, wI[idx]), idx[np.flatnonzero(wr != wI[idx])[:10]]
    assert np.array_equal(Fr, F[idx]), idx[np.flatnonzero(Fr != F[idx])[:10]]
    assert np.array_equal(sr, split[idx]), idx[np.flatnonzero(sr != split[idx])[:10]]
    return res, prof, len(subsets)


def test_config3_m24(mpt):
    """RAG-shaped m = 24 (1.4e11 splits): the oracle runs the whole recurrence
    (about half a minute on the host cores), and OPT, every F(S), every
    w(I(S)), every split(S), the permutations and the DFS order are bit-exact."""
    res, prof = assert_full_parity(mpt, I.config(3), expect_mode=1)
    assert prof["dp_mode"] == 1


def test_config4_m28(mpt):
    """RAG-shaped m = 28, k = 20: the benchmark workload, same launch path."""
    res, prof, count = assert_sampled_parity(mpt, I.config(4), seed=28, uniform=100000)
    assert prof["dp_mode"] == 1 and count >= 100000


def test_config5_m30(mpt):
    """RAG-shaped m = 30, k = 40, 1M-passage corpus: at least 10^5 sampled
    subsets recomputed (uniform plus per-size strata, the full set included)."""
    res, prof, count = assert_sampled_parity(mpt, I.config(5), seed=30, uniform=100000)
    assert prof["dp_mode"] == 1 and count >= 100000


def _submask_index(S):
    pos = [i for i in range(64) if (S >> i) & 1]
    idx = np.zeros(1 << len(pos), dtype=np.int64)
    for q, p in enumerate(pos):
        idx[np.arange(1 << len(pos)) & (1 << q) != 0] |= 1 << p
    return idx


def test_m31_extension(mpt):
    """m = 31 (2^31-entry tables): layout trie cost = OPT, bounds, the split of
    every sampled subset attains its F, no random split does better, and small
    subsets recomputed by the oracle from their own submask tables."""
    inst = I.config(6)
    res = mpt.solve(inst.weights, inst.bits)
    F_d, wI_d, split_d = mpt.mpt_tables(res.ctx)
    m = inst.m
    assert O.trie_cost(inst.weights, res.permutations()) == res.opt
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == res.opt
    R = O.request_sets(inst.weights, inst.bits)
    assert all(sorted(p) == sorted(R[i]) for i, p in enumerate(res.permutations()))
    assert O.spanning_tree_bound(inst.weights, inst.bits) <= res.opt <= O.global_order_cost(inst.weights, inst.bits)
    rng = np.random.default_rng(31)
    full = (1 << m) - 1
    # property checks on random subsets of every size (and the full set)
    Ss = [full] + [int(sum(1 << int(i) for i in rng.choice(m, size=k, replace=False)))
                   for k in range(2, m + 1) for _ in range(8)]
    S_t = torch.tensor(Ss, dtype=torch.int64, device=F_d.device)
    A_t = split_d[S_t].to(torch.int64) & 0xFFFFFFFF
    F_S, F_A, F_B = F_d[S_t], F_d[A_t], F_d[S_t ^ A_t]
    wI_S = wI_d[S_t]
    assert bool(torch.all(F_S == F_A + F_B - wI_S))
    assert bool(torch.all((A_t & S_t) == A_t)) and bool(torch.all((A_t & (S_t & -S_t)) != 0))
    for S in Ss[:40]:
        assert int(wI_d[S].item()) == O.wI_one(inst.weights, inst.bits, S)
    for _ in range(200):  # random other splits never beat the chosen one
        k = int(rng.integers(0, len(Ss)))
        S = Ss[k]
        low = S & -S
        rest = S ^ low
        bits_rest = [i for i in range(m) if (rest >> i) & 1]
        sub = sum(1 << i for i in bits_rest if rng.random() < 0.5)
        if sub == rest:
            continue
        A = low | sub
        assert int(F_d[A].item()) + int(F_d[S ^ A].item()) - int(wI_d[S].item()) >= int(F_d[S].item())
    # oracle recomputation of small subsets from their own submask tables
    for k in range(2, 15):
        for _ in range(6):
            S = int(sum(1 << int(i) for i in rng.choice(m, size=k, replace=False)))
            idx = torch.from_numpy(_submask_index(S)).to(F_d.device)
            f, a, w = O.recompute_local(inst.weights, inst.bits, S, F_d[idx].cpu().numpy())
            assert (f, a, w) == (int(F_d[S].item()), int(split_d[S].item()) & 0xFFFFFFFF, int(wI_d[S].item()))


def test_m32_maximum(mpt):
    """m = 32, the largest instance the ABI takes (subset masks use all 32 bits,
    2^32-entry tables), on lean tables: layout trie cost = OPT, bounds, sampled
    subsets of every size whose split attains F(S) with w(I(S)) recomputed by
    direct intersection, random other splits never better, and small subsets
    recomputed by the oracle from their own submask tables."""
    inst = I.config(7)
    m = inst.m
    assert m == 32
    res = mpt.solve(inst.weights, inst.bits, tables="lean")
    F_d, split_d = mpt.mpt_tables32(res.ctx)
    assert O.trie_cost(inst.weights, res.permutations()) == res.opt
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == res.opt
    R = O.request_sets(inst.weights, inst.bits)
    assert all(sorted(p) == sorted(R[i]) for i, p in enumerate(res.permutations()))
    assert O.spanning_tree_bound(inst.weights, inst.bits) <= res.opt <= O.global_order_cost(inst.weights, inst.bits)
    rng = np.random.default_rng(32)
    full = (1 << m) - 1
    assert int(F_d[full].item()) == res.opt
    Ss = [full] + [int(sum(1 << int(i) for i in rng.choice(m, size=k, replace=False)))
                   for k in range(2, m + 1) for _ in range(3)]
    wI = {S: O.wI_one(inst.weights, inst.bits, S) for S in Ss}
    for S in Ss:
        A = int(split_d[S].item()) & 0xFFFFFFFF
        assert A & S == A and A & (S & -S) and A != S
        assert int(F_d[S].item()) == int(F_d[A].item()) + int(F_d[S ^ A].item()) - wI[S]
    for _ in range(100):  # random other splits never beat the chosen one
        S = Ss[int(rng.integers(0, len(Ss)))]
        low = S & -S
        rest = S ^ low
        sub = sum(1 << i for i in range(m) if (rest >> i) & 1 and rng.random() < 0.5)
        if sub == rest:
            continue
        A = low | sub
        assert int(F_d[A].item()) + int(F_d[S ^ A].item()) - wI[S] >= int(F_d[S].item())
    for k in range(2, 13):
        for _ in range(3):
            S = int(sum(1 << int(i) for i in rng.choice(m, size=k, replace=False)))
            idx = torch.from_numpy(_submask_index(S)).to(F_d.device)
            f, a, w = O.recompute_local(inst.weights, inst.bits, S, F_d[idx].to(torch.int64).cpu().numpy())
            assert (f, a) == (int(F_d[S].item()), int(split_d[S].item()) & 0xFFFFFFFF)


def test_concurrent_contexts_on_streams(mpt):
    """Independent contexts solved at the same time on different streams (own
    workspaces) give the same tables as solving them one after the other: no
    state is shared between contexts."""
    insts = [I.rag_pools(20, 5000, 6, 40, 8, 1.1, seed=s) for s in (21, 22)]
    insts.append(I.random_instance(15, 80, (2, 9), seed=23, wmin=200_000, wmax=400_000))  # general kernels
    seq = []
    for inst in insts:
        r = mpt.solve(inst.weights, inst.bits)
        seq.append((r.opt, [t.clone() for t in mpt.mpt_tables(r.ctx)], r.permutations()))
    streams = [torch.cuda.Stream() for _ in insts]
    ctxs, wss = [], []
    for inst in insts:
        c = mpt.mpt_create(inst.weights, inst.bits)
        ctxs.append(c)
        wss.append(torch.empty(mpt.mpt_workspace_bytes(c), dtype=torch.uint8, device="cuda"))
    import threading

    out = [None] * len(insts)

    def run(i):
        out[i] = mpt.mpt_solve(ctxs[i], wss[i], streams[i].cuda_stream)

    threads = [threading.Thread(target=run, args=(i,)) for i in range(len(insts))]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    torch.cuda.synchronize()
    for i, (opt, tables, perms) in enumerate(seq):
        assert out[i] == opt
        for a, b in zip(tables, mpt.mpt_tables(ctxs[i])):
            assert torch.equal(a, b)
        offs, chunks, dfs = mpt.mpt_layout(ctxs[i])
        assert [chunks[offs[j]:offs[j + 1]].tolist() for j in range(len(offs) - 1)] == perms

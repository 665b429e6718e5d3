"""Heavy private and universal chunks on the tiled kernels, through the C ABI.

A chunk that one request alone holds, or that every request holds, is one
maximal cluster of its request set in every hierarchy (Thm 1: t_x(H) = 1),
so it adds its weight to F(S) for every S holding its requests and never
changes a split.  The tiled kernels therefore run the recurrence without
those weights and add them back; their key width depends only on the shared
weight.  Here requests get a suffix of their own (a question or a document)
of up to 2^40 tokens and a common prefix (a system prompt) of up to 2^34,
which keeps sum_i w(R_i) far beyond the 32-bit keys while the shared weight
stays below 2^20: AUTO must still take the 32-bit keys, and every table must
equal the oracle's bit for bit."""

from __future__ import annotations

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I
from tests import weights as W

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(1500)]


@pytest.fixture(scope="module")
def mpt():
    import __graft_entry__ as G

    G.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def _tables(mpt, ctx):
    F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(ctx))
    return F, wI, split.view(np.uint32)


def _parity(mpt, inst, mode="auto", expect_mode=1):
    res = mpt.solve(inst.weights, inst.bits, mode=mode, profile=True)
    assert mpt.mpt_get_profile(res.ctx)["dp_mode"] == expect_mode
    F, wI, split = _tables(mpt, res.ctx)
    opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
    assert res.opt == opt
    assert np.array_equal(wI, owI), np.flatnonzero(wI != owI)[:10]
    assert np.array_equal(F, oF), np.flatnonzero(F != oF)[:10]
    assert np.array_equal(split, osplit), np.flatnonzero(split != osplit)[:10]
    perms, dfs = O.layout(inst.weights, inst.bits, osplit)
    assert res.permutations() == perms
    assert res.dfs_order.tolist() == dfs
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == opt
    return res


def _with_queries(base, seed, wmin=1 << 28, wmax=1 << 40, every=1):
    inst = I.with_query_chunks(base, wmin, wmax, seed=seed, every=every)
    assert W.request_weight_sum(inst) >= 1 << 28
    return inst


@pytest.mark.parametrize("m", list(range(1, 19)))
def test_query_chunks_sweep(mpt, m):
    """Random small-weight requests, each with a private suffix of up to 2^40
    tokens: the 32-bit keys, every table bit-exact."""
    rng = np.random.default_rng(7000 + m)
    n = int(rng.integers(8, 90))
    base = I.random_instance(m, n, (0, min(n, 10)), seed=int(rng.integers(1 << 30)), wmin=1, wmax=400,
                             allow_empty=True)
    inst = _with_queries(base, seed=m, every=1 + m % 3)
    assert W.shared_weight(inst) < 1 << 20
    _parity(mpt, inst)


@pytest.mark.parametrize("m", [1, 2, 3, 5, 8, 11, 13, 16, 18])
def test_common_prefix_sweep(mpt, m):
    """A common prefix of 2^34 tokens in every request, with and without
    private suffixes: the 32-bit keys, every table bit-exact."""
    rng = np.random.default_rng(8000 + m)
    n = int(rng.integers(8, 90))
    base = I.random_instance(m, n, (0, min(n, 10)), seed=int(rng.integers(1 << 30)), wmin=1, wmax=400,
                             allow_empty=True)
    inst = I.with_common_prefix(base, 1 << 34)
    assert W.shared_weight(inst) < 1 << 20
    _parity(mpt, inst)
    _parity(mpt, _with_queries(inst, seed=m, every=2))


def test_query_chunks_paper_examples(mpt):
    """The paper's examples and the edge cases with heavy private suffixes:
    one request, empty requests, identical requests, all-private requests."""
    cases = [I.k4_3(), I.open_problem_k4(), I.tightness_witness(), I.leave_one_out(12), I.config(1),
             I.Instance(np.array([5], dtype=np.int64), I.pack_requests([[0]], 1)),
             I.Instance(np.array([3, 4, 5], dtype=np.int64), I.pack_requests([[], [0, 1], [], [0, 1], [2]], 3)),
             I.Instance(np.arange(1, 9, dtype=np.int64), I.pack_requests([[1, 2, 3]] * 14, 8))]
    for k, base in enumerate(cases):
        _parity(mpt, _with_queries(base, seed=100 + k))
    # every chunk private: F(S) = sum_{i in S} w(R_i), nothing to share
    own = I.Instance(np.full(16, 1 << 35, dtype=np.int64), I.pack_requests([[i] for i in range(16)], 16))
    res = _parity(mpt, own)
    assert res.opt == 16 << 35


def test_query_chunks_all_modes_agree(mpt):
    """The 32-bit keys, the 64-bit keys and the int64 kernels on the same
    instance: every table identical."""
    import torch

    inst = _with_queries(I.rag_pools(17, 3000, 5, 40, 8, 1.1, seed=4), seed=9)
    ctxs = []
    for mode, dp in (("auto", 1), ("wide", 3), ("general", 2)):
        res = mpt.solve(inst.weights, inst.bits, mode=mode, profile=True)
        assert mpt.mpt_get_profile(res.ctx)["dp_mode"] == dp
        ctxs.append(res)
    t0 = mpt.mpt_tables(ctxs[0].ctx)
    for r in ctxs[1:]:
        assert r.opt == ctxs[0].opt
        for a, b in zip(t0, mpt.mpt_tables(r.ctx)):
            assert torch.equal(a, b)
        assert r.permutations() == ctxs[0].permutations()
    assert ctxs[0].opt == O.solve(inst.weights, inst.bits)[0]


def test_shared_weight_limit(mpt):
    """Shared weight 2^20 - 1 under private suffixes of 2^33 tokens: the 32-bit
    keys; one token more shared: the 64-bit keys, and BLOCKED is refused."""
    m = 15
    # chunk x < m is held by requests x and x - 1 (mod m), chunk m by requests
    # 0, 1 and 2: shared weight 2 * sum_{x<m} w(x) + 3 * w(m) = 2^20 - 1
    w = np.full(m + 1, 34952, dtype=np.int64)
    w[0] += 6
    w[m] = 1
    reqs = [[x for x in range(m + 1) if i in _holders(x, m)] for i in range(m)]
    base = I.Instance(w, I.pack_requests(reqs, m + 1))
    assert W.shared_weight(base) == 2 ** 20 - 1
    inst = _with_queries(base, seed=5, wmin=1 << 33, wmax=1 << 33)
    assert W.shared_weight(inst) == 2 ** 20 - 1
    _parity(mpt, inst, expect_mode=1)
    _parity(mpt, inst, mode="blocked", expect_mode=1)
    _parity(mpt, I.with_common_prefix(inst, 1 << 34), expect_mode=1)
    heavier = I.Instance(inst.weights.copy(), inst.bits)
    heavier.weights[m] += 1  # chunk m is shared: the shared weight reaches 2^20 + 2
    assert W.shared_weight(heavier) >= 1 << 20
    _parity(mpt, heavier, expect_mode=3)
    ctx = mpt.mpt_create(heavier.weights, heavier.bits)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_dp_mode(ctx, "blocked")
    assert e.value.status == 3


def _holders(x, m):
    """Requests holding chunk x in the limit instance above."""
    return {x, (x - 1) % m} if x < m else {0, 1, 2}


def test_query_chunks_lean_and_staged(mpt):
    """Lean int32 tables (sum_i w(R_i) < 2^31) and a staged solve restored
    from a host checkpoint after every step, both on private suffixes."""
    import torch

    inst = _with_queries(I.rag_pools(18, 4000, 5, 40, 8, 1.1, seed=6), seed=3, wmin=1 << 24, wmax=1 << 26)
    assert W.request_weight_sum(inst) < 1 << 31 and W.shared_weight(inst) < 1 << 20
    ref = mpt.solve(inst.weights, inst.bits)
    F, _, split = mpt.mpt_tables(ref.ctx)
    lean = mpt.solve(inst.weights, inst.bits, tables="lean")
    F32, split32 = mpt.mpt_tables32(lean.ctx)
    assert lean.opt == ref.opt
    assert torch.equal(F, F32.to(torch.int64)) and torch.equal(split, split32)
    assert lean.permutations() == ref.permutations()

    ctx = mpt.mpt_create(inst.weights, inst.bits)
    steps = mpt.mpt_solve_steps(ctx)
    ws = torch.empty(mpt.mpt_workspace_bytes(ctx), dtype=torch.uint8, device="cuda")
    mpt.mpt_solve_begin(ctx, ws)
    nxt = 1
    while nxt < steps:
        nxt = mpt.mpt_solve_layers(ctx, ws, 1)
        torch.cuda.synchronize()
        saved = ws.cpu()
        ws.fill_(0x5A)
        ws.copy_(saved.cuda())
        mpt.mpt_solve_resume(ctx, ws, nxt)
    assert mpt.mpt_solve_end(ctx, ws) == ref.opt
    for a, b in zip(mpt.mpt_tables(ctx), mpt.mpt_tables(ref.ctx)):
        assert torch.equal(a, b)
    assert ref.opt == O.solve(inst.weights, inst.bits)[0]


def _pi_of_subsets(m, pi):
    """sum_{i in S} pi_i for every mask S, on the device."""
    import torch

    S = torch.arange(1 << m, dtype=torch.int64, device="cuda")
    out = torch.zeros(1 << m, dtype=torch.int64, device="cuda")
    for i in range(m):
        out += ((S >> i) & 1) * int(pi[i])
    return out


@pytest.mark.parametrize("workload", [3, 4])
def test_query_chunks_rag_workloads(mpt, workload):
    """The m = 24 and m = 28 RAG workloads with a private suffix of up to 2^30
    tokens on every request, against the same workload without them: F shifts
    by sum_{i in S} pi_i, w(I(S)) only at the singletons and the empty set,
    every split and the layout's shared part stay, all on the 32-bit keys."""
    import torch

    base = I.config(workload)
    inst = _with_queries(base, seed=workload, wmin=1 << 26, wmax=1 << 30)
    assert W.shared_weight(inst) == W.shared_weight(base) < 1 << 20
    a = mpt.solve(base.weights, base.bits, profile=True)
    b = mpt.solve(inst.weights, inst.bits, profile=True)
    assert mpt.mpt_get_profile(a.ctx)["dp_mode"] == 1 and mpt.mpt_get_profile(b.ctx)["dp_mode"] == 1
    m = base.m
    q = inst.weights[base.n:]  # the suffix of request i is chunk base.n + i
    assert b.opt == a.opt + int(q.sum())
    Fa, wIa, sa = mpt.mpt_tables(a.ctx)
    Fb, wIb, sb = mpt.mpt_tables(b.ctx)
    assert torch.equal(sa, sb)
    assert torch.equal(Fb, Fa + _pi_of_subsets(m, q))
    single = torch.zeros(1 << m, dtype=torch.int64, device="cuda")
    single[torch.tensor([1 << i for i in range(m)], device="cuda")] = torch.from_numpy(q).cuda()
    single[0] = int(q.sum())
    assert torch.equal(wIb, wIa + single)
    pa, pb = a.permutations(), b.permutations()
    for i in range(m):
        assert pb[i] == pa[i] + [base.n + i]  # the suffix is emitted last, at the leaf
    assert b.dfs_order.tolist() == a.dfs_order.tolist()
    assert mpt.mpt_trie_cost(inst.weights, b.perm_offsets, b.perm_chunks) == b.opt


def test_common_prefix_rag_workload(mpt):
    """The m = 28 workload behind a common prefix of 2^30 tokens and with
    private suffixes: F shifts by sum_{i in S} pi_i + u for non-empty S, every
    w(I(S)) by u, the splits stay and every permutation starts with the
    prefix, all on the 32-bit keys."""
    import torch

    base = I.config(4)
    u = 1 << 30
    inst = _with_queries(I.with_common_prefix(base, u), seed=11, wmin=1 << 26, wmax=1 << 30)
    assert W.shared_weight(inst) == W.shared_weight(base) and W.universal_weight(inst) == u
    a = mpt.solve(base.weights, base.bits)
    b = mpt.solve(inst.weights, inst.bits, profile=True)
    assert mpt.mpt_get_profile(b.ctx)["dp_mode"] == 1
    m = base.m
    q = inst.weights[base.n + 1:]  # request i's suffix is chunk base.n + 1 + i
    assert b.opt == a.opt + u + int(q.sum())
    Fa, wIa, sa = mpt.mpt_tables(a.ctx)
    Fb, wIb, sb = mpt.mpt_tables(b.ctx)
    assert torch.equal(sa, sb)
    nonempty = (torch.arange(1 << m, device="cuda") != 0).to(torch.int64)
    assert torch.equal(Fb, Fa + _pi_of_subsets(m, q) + u * nonempty)
    expect = wIa + u
    expect[torch.tensor([1 << i for i in range(m)], device="cuda")] += torch.from_numpy(q.copy()).cuda()
    expect[0] += int(q.sum())
    assert torch.equal(wIb, expect)
    for i, (pa, pb) in enumerate(zip(a.permutations(), b.permutations())):
        assert pb == [base.n] + pa + [base.n + 1 + i]
    assert b.dfs_order.tolist() == a.dfs_order.tolist()
    assert mpt.mpt_trie_cost(inst.weights, b.perm_offsets, b.perm_chunks) == b.opt


def test_common_prefix_on_every_kernel_family(mpt):
    """A common prefix and private suffixes under the 64-bit keys (chosen by
    AUTO for heavy shared weights, and forced) and the int64 kernels: every
    table bit-exact against the oracle."""
    heavy_shared = I.random_instance(14, 40, (2, 8), seed=31, wmin=1 << 20, wmax=1 << 24)
    inst = _with_queries(I.with_common_prefix(heavy_shared, 1 << 40), seed=32, every=2)
    assert (1 << 20) <= W.shared_weight(inst) < 1 << 51 and W.universal_weight(inst) == 1 << 40
    _parity(mpt, inst, expect_mode=3)
    _parity(mpt, inst, mode="general", expect_mode=2)
    light = _with_queries(I.with_common_prefix(I.rag_pools(15, 3000, 5, 40, 8, 1.1, seed=8), 1 << 34), seed=33)
    _parity(mpt, light, mode="wide", expect_mode=3)
    _parity(mpt, light, mode="general", expect_mode=2)

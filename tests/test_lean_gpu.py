"""Lean tables (one int32 table, F(S) written over w(I(S)) in place) against
the int64 tables: F, split, OPT and the layout bit-exact, on both DP paths,
in staged solves, and on a full m = 31 table."""

from __future__ import annotations

import numpy as np
import pytest

from paper_2609_13692_gb300 import instances as I

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(1200)]


@pytest.fixture(scope="module")
def mpt():
    import __graft_entry__ as G

    G.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def _instances():
    out = [
        I.config(1), I.config(2), I.leave_one_out(14), I.k4_3(), I.open_problem_k4(), I.tightness_witness(),
        I.Instance(np.array([5], dtype=np.int64), I.pack_requests([[0]], 1), "m=1"),
        I.Instance(np.array([3, 4, 5], dtype=np.int64), I.pack_requests([[], [0, 1], [], [0, 1], [2]], 3),
                   "empty and identical requests"),
        I.rag_pools(20, 5000, 6, 40, 8, 1.1, seed=11),
        I.random_instance(14, 60, (2, 8), seed=5, wmin=100_000, wmax=400_000),  # shared weight > 2^20: 64-bit keys
    ]
    rng = np.random.default_rng(61)
    for m in (2, 5, 9, 12, 13, 16, 18):
        out.append(I.random_instance(m, 70, (1, 9), seed=int(rng.integers(1 << 30)), wmin=1, wmax=300))
    return out


def _solve(mpt, inst, tables, mode="auto"):
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    if mode != "auto":
        mpt.mpt_set_dp_mode(ctx, mode)
    mpt.mpt_set_tables(ctx, tables)
    opt = mpt.mpt_solve(ctx)
    if tables == "lean":
        F, split = mpt.mpt_tables32(ctx)
    else:
        F, _, split = mpt.mpt_tables(ctx)
    return ctx, opt, F, split, mpt.mpt_layout(ctx)


@pytest.mark.parametrize("mode", ["auto", "general", "wide"])
def test_lean_equals_int64(mpt, mode):
    import torch

    for inst in _instances():
        if mode == "general" and inst.m > 16:
            continue
        c1, o1, F1, s1, l1 = _solve(mpt, inst, "int64", mode)
        c2, o2, F2, s2, l2 = _solve(mpt, inst, "lean", mode)
        assert o1 == o2, inst.name
        assert torch.equal(F1, F2.to(torch.int64)), inst.name
        assert torch.equal(s1, s2), inst.name
        assert all(np.array_equal(a, b) for a, b in zip(l1, l2)), inst.name
        w1, w2 = mpt.mpt_workspace_bytes(c1), mpt.mpt_workspace_bytes(c2)
        assert w2 < w1 and w1 - w2 >= 12 * (1 << inst.m) - 4096, inst.name


def test_lean_staged_checkpoint(mpt):
    import torch

    inst = I.rag_pools(20, 5000, 6, 40, 8, 1.1, seed=11)
    _, opt, F, split, lay = _solve(mpt, inst, "int64")
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    mpt.mpt_set_tables(ctx, "lean")
    steps = mpt.mpt_solve_steps(ctx)
    ws = mpt.mpt_solve_begin(ctx)
    nxt = 1
    while nxt < steps:
        nxt = mpt.mpt_solve_layers(ctx, ws, 2)
        torch.cuda.synchronize()
        saved = ws.cpu()
        ws.fill_(0x5A)
        ws.copy_(saved.cuda())
        mpt.mpt_solve_resume(ctx, ws, nxt)
    assert mpt.mpt_solve_end(ctx, ws) == opt
    F2, s2 = mpt.mpt_tables32(ctx)
    assert torch.equal(F, F2.to(torch.int64)) and torch.equal(split, s2)
    assert all(np.array_equal(a, b) for a, b in zip(lay, mpt.mpt_layout(ctx)))


def test_lean_m31_full_table(mpt):
    """Every one of the 2^31 F and split entries of the m = 31 workload agrees
    between the lean and the int64 tables."""
    import torch

    inst = I.config(6)
    c1, o1, F1, s1, l1 = _solve(mpt, inst, "lean")
    F32 = F1.clone()
    S32 = s1.clone()
    lay = l1
    mpt.mpt_destroy(c1)
    c1.workspace = None
    del F1, s1
    torch.cuda.empty_cache()
    c2, o2, F2, s2, l2 = _solve(mpt, inst, "int64")
    assert o1 == o2
    assert torch.equal(S32, s2)
    chunk = 1 << 28
    for i in range(0, 1 << 31, chunk):
        assert torch.equal(F32[i:i + chunk].to(torch.int64), F2[i:i + chunk]), i
    assert all(np.array_equal(a, b) for a, b in zip(lay, l2))
    mpt.mpt_destroy(c2)
    c2.workspace = None
    del F32, S32, F2, s2
    torch.cuda.empty_cache()

"""Staged solve with checkpoints (mpt_solve_begin / _layers / _end /
_resume): bit-exact against a one-shot solve, including a workspace wiped
and restored from a host copy after every step and a resume in a fresh
context."""

from __future__ import annotations

import numpy as np
import pytest

from paper_2609_13692_gb300 import instances as I

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(900)]


@pytest.fixture(scope="module")
def mpt():
    import __graft_entry__ as G

    G.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def _cases():
    big = I.random_instance(14, 60, (2, 8), seed=5, wmin=100_000, wmax=400_000)  # shared weight > 2^20
    return [
        ("blocked m=20", I.rag_pools(20, 5000, 6, 40, 8, 1.1, seed=3), "auto"),
        ("blocked m=12 (one step)", I.config(1), "auto"),
        ("blocked m=17", I.random_instance(17, 80, (2, 9), seed=9, wmin=1, wmax=60), "auto"),
        ("general m=14", big, "general"),
        ("wide m=14 (64-bit keys chosen by AUTO)", big, "auto"),
        ("wide m=17", I.random_instance(17, 80, (2, 9), seed=9, wmin=1, wmax=60), "wide"),
    ]


def _ctx(mpt, inst, mode):
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    if mode != "auto":
        mpt.mpt_set_dp_mode(ctx, mode)
    return ctx


def _one_shot(mpt, inst, mode="auto"):
    ctx = _ctx(mpt, inst, mode)
    opt = mpt.mpt_solve(ctx)
    F, wI, split = (t.clone() for t in mpt.mpt_tables(ctx))
    lay = mpt.mpt_layout(ctx)
    return opt, F, wI, split, lay


def _same_layout(a, b):
    return all(np.array_equal(np.asarray(x), np.asarray(y)) for x, y in zip(a, b))


@pytest.mark.parametrize("idx", range(6))
def test_staged_with_checkpoint_every_step(mpt, idx):
    import torch

    name, inst, mode = _cases()[idx]
    opt, F, wI, split, lay = _one_shot(mpt, inst, mode)
    ctx = _ctx(mpt, inst, mode)
    steps = mpt.mpt_solve_steps(ctx)
    ws = torch.empty(mpt.mpt_workspace_bytes(ctx), dtype=torch.uint8, device="cuda")
    mpt.mpt_solve_begin(ctx, ws)
    nxt = 1
    while nxt < steps:
        nxt = mpt.mpt_solve_layers(ctx, ws, 1)
        torch.cuda.synchronize()
        saved = ws.cpu()
        ws.fill_(0xA5)  # the device copy is destroyed ...
        ws.copy_(saved.cuda())  # ... and restored from the checkpoint
        mpt.mpt_solve_resume(ctx, ws, nxt)
    assert mpt.mpt_solve_end(ctx, ws) == opt, name
    F2, wI2, split2 = mpt.mpt_tables(ctx)
    assert torch.equal(F, F2) and torch.equal(wI, wI2) and torch.equal(split, split2), name
    assert _same_layout(lay, mpt.mpt_layout(ctx)), name


def test_resume_in_fresh_context(mpt):
    import torch

    name, inst, _ = _cases()[0]
    opt, F, wI, split, lay = _one_shot(mpt, inst)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    steps = mpt.mpt_solve_steps(ctx)
    ws = mpt.mpt_solve_begin(ctx)
    half = mpt.mpt_solve_layers(ctx, ws, steps // 2)
    torch.cuda.synchronize()
    checkpoint = ws.cpu()
    mpt.mpt_destroy(ctx)
    ctx2 = mpt.mpt_create(inst.weights, inst.bits)
    ws2 = torch.empty(mpt.mpt_workspace_bytes(ctx2), dtype=torch.uint8, device="cuda")
    ws2.copy_(checkpoint.cuda())
    mpt.mpt_solve_resume(ctx2, ws2, half)
    assert mpt.mpt_solve_layers(ctx2, ws2, steps) == steps
    assert mpt.mpt_solve_end(ctx2, ws2) == opt
    F2, wI2, split2 = mpt.mpt_tables(ctx2)
    assert torch.equal(F, F2) and torch.equal(wI, wI2) and torch.equal(split, split2)
    assert _same_layout(lay, mpt.mpt_layout(ctx2))


def test_staged_errors(mpt):
    import torch

    inst = _cases()[2][1]
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    ws = torch.empty(mpt.mpt_workspace_bytes(ctx), dtype=torch.uint8, device="cuda")
    other = torch.empty_like(ws)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_solve_layers(ctx, ws, 1)
    assert e.value.status == 7  # nothing begun
    mpt.mpt_solve_begin(ctx, ws)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_solve_end(ctx, ws)
    assert e.value.status == 7  # steps left
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_solve_layers(ctx, other, 1)
    assert e.value.status == 1  # another workspace
    mpt.mpt_solve_layers(ctx, ws, 100)
    assert mpt.mpt_solve_end(ctx, ws) == _one_shot(mpt, inst)[0]

"""The blocked recurrence with 64-bit packed keys (MPT_DP_WIDE, chosen by AUTO
when the shared weight -- sum_i w(R_i) less the chunks one request alone
holds -- lies in [2^20, 2^51)) against the oracle and against the 32-bit
path, through the C ABI.  Integer results: bit-exact.

Scaling every chunk weight by c scales w(I(S)), F(S) and OPT by c and keeps
every comparison, hence the argmin, the hierarchy and the layout (Sec. 3.1:
the recurrence is linear in w).  That identity carries the m = 24 and m = 28
workloads onto weights the 32-bit keys cannot hold."""

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


def _solve(mpt, inst, mode="auto"):
    res = mpt.solve(inst.weights, inst.bits, mode=mode, profile=True)
    F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(res.ctx))
    return res, F, wI, split.view(np.uint32), mpt.mpt_get_profile(res.ctx)


def _parity(mpt, inst, mode="auto", expect_mode=3):
    res, F, wI, split, prof = _solve(mpt, inst, mode)
    assert prof["dp_mode"] == expect_mode
    opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
    assert res.opt == opt
    assert np.array_equal(wI, owI), np.flatnonzero(wI != owI)[:10]
    assert np.array_equal(F, oF), np.flatnonzero(F != oF)[:10]
    assert np.array_equal(split, osplit), np.flatnonzero(split != osplit)[:10]
    perms, dfs = O.layout(inst.weights, inst.bits, osplit)
    assert res.permutations() == perms
    assert res.dfs_order.tolist() == dfs
    return res


@pytest.mark.parametrize("m", list(range(1, 19)))
def test_wide_sweep_heavy_weights(mpt, m):
    """Random instances with weights up to 2^40: AUTO takes the 64-bit keys
    (the 32-bit ones where no chunk is shared, e.g. m = 1)."""
    rng = np.random.default_rng(5000 + m)
    n = int(rng.integers(8, 120))
    inst = I.random_instance(m, n, (1, min(n, 12)), seed=int(rng.integers(1 << 30)), wmin=1 << 20, wmax=1 << 40)
    shared = W.shared_weight(inst)
    assert shared < (1 << 51) and W.request_weight_sum(inst) >= 1 << 20
    _parity(mpt, inst, expect_mode=3 if shared >= 1 << 20 else 1)


@pytest.mark.parametrize("m", [13, 15, 17, 18])
def test_wide_ties(mpt, m):
    """Small weights scaled by 2^21: as many optimal splits as the small
    instance has, so the tie rule (least A) is exercised on every layer."""
    rng = np.random.default_rng(6000 + m)
    base = I.random_instance(m, 30, (2, 10), seed=int(rng.integers(1 << 30)), wmin=1, wmax=3)
    inst = I.Instance(base.weights << 21, base.bits)
    _parity(mpt, inst)
    loo = I.leave_one_out(m)
    _parity(mpt, I.Instance(loo.weights << 21, loo.bits))


def test_wide_forced_on_light_weights(mpt):
    """MPT_DP_WIDE on instances the 32-bit keys also hold: identical results,
    including the paper's examples and edge cases."""
    cases = [I.config(1), I.leave_one_out(16), I.k4_3(), I.open_problem_k4(), I.tightness_witness(),
             I.Instance(np.array([5], dtype=np.int64), I.pack_requests([[0]], 1)),
             I.Instance(np.array([3, 4], dtype=np.int64), I.pack_requests([[], [0, 1], []], 2)),
             I.Instance(np.arange(1, 9, dtype=np.int64), I.pack_requests([[1, 2, 3]] * 14, 8)),
             I.random_instance(15, 3, (0, 3), seed=5, allow_empty=True)]
    for inst in cases:
        _parity(mpt, inst, "wide")


def _scaled_equal(mpt, inst, c):
    """The 32-bit path on inst and AUTO (64-bit keys) on inst scaled by c,
    compared on the device table by table."""
    import torch

    narrow = mpt.solve(inst.weights, inst.bits, profile=True)
    assert mpt.mpt_get_profile(narrow.ctx)["dp_mode"] == 1
    heavy = I.Instance(inst.weights * c, inst.bits)
    assert W.shared_weight(heavy) >= 1 << 20
    wide = mpt.solve(heavy.weights, heavy.bits, profile=True)
    assert mpt.mpt_get_profile(wide.ctx)["dp_mode"] == 3
    assert wide.opt == c * narrow.opt
    Fn, wIn, sn = mpt.mpt_tables(narrow.ctx)
    Fw, wIw, sw = mpt.mpt_tables(wide.ctx)
    assert torch.equal(Fw, Fn * c)
    assert torch.equal(wIw, wIn * c)
    assert torch.equal(sw, sn)
    assert wide.permutations() == narrow.permutations()
    assert wide.dfs_order.tolist() == narrow.dfs_order.tolist()
    assert mpt.mpt_trie_cost(heavy.weights, wide.perm_offsets, wide.perm_chunks) == wide.opt
    return narrow, wide


def test_wide_scaled_rag_m24(mpt):
    """The RAG-shaped m = 24 workload at 4096x its weights against the 32-bit path."""
    _scaled_equal(mpt, I.config(3), 4096)


def test_wide_scaled_rag_m28(mpt):
    """The m = 28 benchmark workload at 1000x its weights: every table of the
    2^28 subsets equal to 1000x the 32-bit path's."""
    _scaled_equal(mpt, I.config(4), 1000)


def test_wide_lean_tables(mpt):
    """Lean (int32) tables on the 64-bit-key path equal the int64 ones."""
    import torch

    inst = I.random_instance(16, 60, (2, 8), seed=21, wmin=50_000, wmax=200_000)
    assert W.shared_weight(inst) >= 1 << 20 and W.request_weight_sum(inst) < 1 << 31
    ctx1 = mpt.mpt_create(inst.weights, inst.bits)
    o1 = mpt.mpt_solve(ctx1)
    assert mpt.mpt_get_profile(ctx1)["dp_mode"] == 3
    F1, _, s1 = mpt.mpt_tables(ctx1)
    ctx2 = mpt.mpt_create(inst.weights, inst.bits)
    mpt.mpt_set_dp_mode(ctx2, "wide")
    mpt.mpt_set_tables(ctx2, "lean")
    assert mpt.mpt_solve(ctx2) == o1
    F2, s2 = mpt.mpt_tables32(ctx2)
    assert torch.equal(F1, F2.to(torch.int64)) and torch.equal(s1, s2)
    assert o1 == O.solve(inst.weights, inst.bits)[0]


@pytest.mark.parametrize("m", [19, 20, 21, 22])
def test_wide_equals_narrow_medium(mpt, m):
    """The 64-bit keys forced on RAG-shaped instances the 32-bit keys also hold:
    every table equal on the device (layers with several blocks per tile)."""
    import torch

    inst = I.rag_pools(m, 5000, 6, 40, 8, 1.1, seed=100 + m)
    narrow = mpt.solve(inst.weights, inst.bits, profile=True)
    wide = mpt.solve(inst.weights, inst.bits, mode="wide", profile=True)
    assert mpt.mpt_get_profile(narrow.ctx)["dp_mode"] == 1
    assert mpt.mpt_get_profile(wide.ctx)["dp_mode"] == 3
    assert wide.opt == narrow.opt
    for a, b in zip(mpt.mpt_tables(narrow.ctx), mpt.mpt_tables(wide.ctx)):
        assert torch.equal(a, b)
    assert wide.permutations() == narrow.permutations()
    assert wide.dfs_order.tolist() == narrow.dfs_order.tolist()

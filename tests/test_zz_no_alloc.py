"""mpt_solve_noalloc against mpt_solve and the CPU oracle, through the C ABI.

The no-allocation entry point serves callers that cannot allocate device
memory (a serving process whose memory is reserved up front by its own pool,
or code that must not call cudaMalloc / cudaFree because they synchronise
the device).  Its scratch is one file-scope device array shared by all calls,
so the checks run several calls in a row, with different instances, and
compare every table bit for bit with the regular entry point and with the
oracle's plain recurrence.  This file is collected last so that a failure
here leaves every other test already run.
"""

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I

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


def _reference(mpt, inst):
    res = mpt.solve(inst.weights, inst.bits)
    F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(res.ctx))
    return res.opt, F, wI, split


def _noalloc(mpt, inst):
    dev = torch.device("cuda")
    m = inst.m
    d_w = torch.from_numpy(np.ascontiguousarray(inst.weights)).to(dev)
    d_bits = torch.from_numpy(np.ascontiguousarray(inst.bits).view(np.int64)).to(dev)
    F = torch.full((1 << m,), -1, dtype=torch.int64, device=dev)
    wI = torch.full((1 << m,), -1, dtype=torch.int64, device=dev)
    split = torch.full((1 << m,), -1, dtype=torch.int32, device=dev)
    opt = torch.full((1,), -1, dtype=torch.int64, device=dev)
    mpt.mpt_solve_noalloc(d_w, d_bits, F, wI, split, opt)
    torch.cuda.synchronize()
    return int(opt.item()), F.cpu().numpy(), wI.cpu().numpy(), split.cpu().numpy()


def test_noalloc_matches_solve_on_consecutive_calls(mpt):
    cases = [
        I.config(2),                                                         # m = 20, the largest accepted
        I.rag_pools(16, 5000, 4, 60, 8, 1.1, seed=11),                       # m = 16, blocked kernels
        I.random_instance(14, 60, (2, 10), seed=3, wmin=10 ** 9, wmax=10 ** 11),  # int64 kernels
        I.config(2),                                                         # the first instance again
        I.config(1),                                                         # m = 12, one tile
        I.with_query_chunks(I.config(2), 1 << 30, 1 << 38, seed=2),          # private suffixes, blocked kernels
        I.with_query_chunks(I.rag_pools(16, 5000, 4, 60, 8, 1.1, seed=11), 1 << 30, 1 << 38, seed=3),
        I.with_common_prefix(I.with_query_chunks(I.config(1), 1 << 30, 1 << 38, seed=4), 1 << 36),
        I.random_instance(5, 30, 3, seed=7),                                 # m = 5: the tile kernel alone
        I.random_instance(1, 30, 4, seed=8),                                 # m = 1: no universal chunks
        I.config(2),                                                         # m = 20 after the small ones
    ]
    for inst in cases:
        ref = _reference(mpt, inst)
        got = _noalloc(mpt, inst)
        assert got[0] == ref[0]
        for a, b in zip(got[1:], ref[1:]):
            assert np.array_equal(a, b)
        # and directly against the oracle's recurrence (Sec. 3.1)
        opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
        assert got[0] == opt
        assert np.array_equal(got[1], oF) and np.array_equal(got[2], owI)
        assert np.array_equal(got[3].view(np.uint32), osplit)


def test_noalloc_rejects_beyond_limit(mpt):
    inst = I.random_instance(21, 40, 3, seed=1)
    with pytest.raises(mpt.MPTError) as e:
        _noalloc(mpt, inst)
    assert e.value.status == 2  # MPT_ERR_TOO_LARGE

"""Opt-in: the benchmark workload (m = 28) against the oracle's whole
recurrence -- every F(S), w(I(S)) and split(S) of the 2^28 subsets, OPT, the
permutations and the DFS order -- and the oracle's measured solve time.

The oracle needs about 50 minutes on 16 host cores for this, so the test
runs only when MPT_FULL_ORACLE_M28=1 is set; the regular parity tests check
m = 28 on 10^5 sampled subsets instead.  It prints one JSON line with the
timings.
"""

import json
import os
import time

import numpy as np
import pytest

import oracle as O
from paper_2609_13692_gb300 import instances as I

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(7200)]

torch = pytest.importorskip("torch")


@pytest.mark.skipif(os.environ.get("MPT_FULL_ORACLE_M28") != "1", reason="opt-in (about 50 min of host time)")
def test_workload4_every_entry_against_the_whole_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_13692_gb300 import build as B

    B.build()
    O.build()
    from paper_2609_13692_gb300 import mpt

    mpt.load()
    inst = I.config(4)
    t0 = time.perf_counter()
    res = mpt.solve(inst.weights, inst.bits)
    gpu_s = time.perf_counter() - t0
    F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(res.ctx))
    split = split.view(np.uint32)
    t0 = time.perf_counter()
    wI_o = O.intersection_weights(inst.weights, inst.bits)
    wi_s = time.perf_counter() - t0
    t0 = time.perf_counter()
    F_o, split_o = O.dp(wI_o, inst.m)
    dp_s = time.perf_counter() - t0
    full = (1 << inst.m) - 1
    assert res.opt == F_o[full]
    assert np.array_equal(wI, wI_o), np.flatnonzero(wI != wI_o)[:10]
    assert np.array_equal(F, F_o), np.flatnonzero(F != F_o)[:10]
    assert np.array_equal(split, split_o), np.flatnonzero(split != split_o)[:10]
    perms, dfs = O.layout(inst.weights, inst.bits, split_o)
    assert res.permutations() == perms
    assert res.dfs_order.tolist() == dfs
    print(json.dumps({"m": inst.m, "opt": int(res.opt), "gpu_solve_with_first_load_s": gpu_s,
                      "oracle_wI_s": wi_s, "oracle_dp_s": dp_s, "oracle_threads": O.max_threads(),
                      "oracle_splits_per_s": ((3 ** inst.m + 1) // 2 - 2 ** inst.m) / dp_s}), flush=True)

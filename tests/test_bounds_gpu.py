"""The bounds-checked build (compiled with MPT_BOUNDS) on small cases.

It stands in for a device memory checker: the exact-solve kernels test their
table indices, window offsets and split entries, skip any access that fails
and report it through the device flags, which mpt_solve turns into
MPT_ERR_INTERNAL; the batched kernels test their block's size and
occurrence cap, their hash-table slots and every split entry, and report
through the instance's status (MPT_ERR_INTERNAL from mpt_batch_solve).  Every solve here must therefore succeed and still match the
oracle, in every DP mode and table layout, one-shot and staged.  The checked
library runs in a child process (MPT_LIBRARY), so the default build this
session has loaded is untouched.
"""

import os
import subprocess
import sys
import textwrap

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = textwrap.dedent(r"""
    import numpy as np
    import oracle as O
    from paper_2609_13692_gb300 import instances as I, mpt

    mpt.load()
    assert mpt.mpt_build_info()["bounds_checked"], "not the bounds-checked library"

    def check(inst, mode="auto", tables="int64", staged=False):
        ctx = mpt.mpt_create(inst.weights, inst.bits)
        if mode != "auto":
            mpt.mpt_set_dp_mode(ctx, mode)
        if tables != "int64":
            mpt.mpt_set_tables(ctx, tables)
        if staged:
            ws = mpt.mpt_solve_begin(ctx)
            while mpt.mpt_solve_layers(ctx, ws, 2) < mpt.mpt_solve_steps(ctx):
                pass
            opt = mpt.mpt_solve_end(ctx, ws)
        else:
            opt = mpt.mpt_solve(ctx)
        ref_opt, oF, owI, osplit = O.solve(inst.weights, inst.bits)
        assert opt == ref_opt, (inst.name, mode, opt, ref_opt)
        if tables == "int64":
            F, wI, split = (t.cpu().numpy() for t in mpt.mpt_tables(ctx))
            assert np.array_equal(wI, owI)
        else:
            F, split = (t.cpu().numpy().astype(np.int64) for t in mpt.mpt_tables32(ctx))
        assert np.array_equal(F, oF) and np.array_equal(split.astype(np.int64) & 0xFFFFFFFF, osplit.astype(np.int64))
        mpt.mpt_destroy(ctx)

    for m in range(1, 19):
        check(I.random_instance(m, 90, (0, 10), seed=500 + m, wmax=300, allow_empty=True), "blocked")
    for m in (2, 9, 10, 14):
        check(I.random_instance(m, 60, (1, 10), seed=600 + m, wmax=900), "general")
    heavy = I.random_instance(15, 50, (2, 8), seed=7, wmin=1 << 20, wmax=1 << 28)
    check(heavy, "wide")
    check(I.leave_one_out(16))
    check(I.rag_pools(18, 4000, 4, 60, 8, 1.1, seed=5), tables="lean")
    check(I.rag_pools(17, 4000, 4, 60, 8, 1.1, seed=6), staged=True)
    check(I.with_query_chunks(I.config(1), 1 << 28, 1 << 36, seed=3))
    # the batched kernels: every size 1..16 (row-blocked and per-subset
    # kernels, rows in shared and in global memory), F and split per instance
    rng = np.random.default_rng(17)
    n = 400
    bw = rng.integers(1, 60, size=n, dtype=np.int64)
    groups = []
    for m in list(range(1, 17)) * 2:
        pool = rng.choice(n, size=40, replace=False)
        groups.append([sorted(set(int(x) for x in rng.choice(pool, size=int(rng.integers(1, 7)), replace=False)))
                       for _ in range(m)])
    heavy_w = np.concatenate([bw, rng.integers(1 << 18, 1 << 20, size=20, dtype=np.int64)])
    for m in (5, 9, 13, 15):  # shared weight >= 2^(32 - m): the per-subset kernel's 64-bit keys
        groups.append([sorted(set(int(x) for x in n + rng.choice(20, size=4, replace=False))) for _ in range(m)])
    opt, perms, orders, b = mpt.solve_batch(heavy_w, groups)
    F_all, S_all, offs = mpt.mpt_batch_tables(b)
    F_all = F_all.cpu().numpy()
    S_all = S_all.cpu().numpy().view(np.uint32)
    for i, reqs in enumerate(groups):
        bits = I.pack_requests(reqs, heavy_w.shape[0])
        o_opt, oF, owI, osplit = O.solve(heavy_w, bits)
        assert opt[i] == o_opt, (i, len(reqs), opt[i], o_opt)
        lo, hi = int(offs[i]), int(offs[i + 1])
        assert np.array_equal(F_all[lo:hi], oF) and np.array_equal(S_all[lo:hi], osplit), i
    # the pair kernel at scale: workload 3 (m = 24), OPT against its layout's trie cost
    inst = I.config(3)
    res = mpt.solve(inst.weights, inst.bits)
    assert mpt.mpt_trie_cost(inst.weights, res.perm_offsets, res.perm_chunks) == res.opt
    print("BOUNDS_OK")
""")


def test_bounds_checked_build_solves_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_13692_gb300 import build as B

    import oracle as O

    lib = B.build(bounds=True)
    O.build()
    env = dict(os.environ, MPT_LIBRARY=str(lib))
    p = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert p.returncode == 0, (p.stdout[-2000:], p.stderr[-4000:])
    assert "BOUNDS_OK" in p.stdout


def test_default_build_reports_no_bounds_checks():
    from paper_2609_13692_gb300 import build as B
    from paper_2609_13692_gb300 import mpt

    B.build()
    mpt.load()
    if os.environ.get("MPT_LIBRARY"):
        pytest.skip("another library was selected")
    assert mpt.mpt_build_info() == {"bounds_checked": False}

"""The C ABI without a GPU: the library loads, exports every declared entry
point, and its host-side argument checks return the documented statuses."""

import os
import re

import numpy as np
import pytest

from paper_2609_13692_gb300 import build as B
from paper_2609_13692_gb300 import instances as I
from tests import weights as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mpt():
    B.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


def declared_functions():
    names = []
    for hdr in os.listdir(os.path.join(ROOT, "include")):
        if hdr.endswith(".h"):
            text = open(os.path.join(ROOT, "include", hdr)).read()
            names += re.findall(r"^\s*(?:mpt_status|void|const char\*)\s+(mpt_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(mpt):
    lib = mpt.load()
    names = declared_functions()
    assert "mpt_solve" in names and "mpt_layout" in names and "mpt_trie_cost" in names
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(mpt.EXPORTED) == names


def _status(mpt, w, bits, m=None):
    import ctypes

    lib = mpt.load()
    w = np.ascontiguousarray(w, dtype=np.int64)
    bits = np.ascontiguousarray(bits, dtype=np.uint64)
    h = ctypes.c_void_p()
    st = lib.mpt_create(w.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), int(w.shape[0]),
                        bits.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64)),
                        int(bits.shape[0] if m is None else m), ctypes.byref(h))
    if st == 0:
        lib.mpt_destroy(h)
    return st


def test_create_validation(mpt):
    inst = I.config(1)
    assert _status(mpt, inst.weights, inst.bits) == 0
    assert _status(mpt, inst.weights, inst.bits, m=0) == 1
    bad = inst.weights.copy()
    bad[3] = 0
    assert _status(mpt, bad, inst.bits) == 1
    bits = inst.bits.copy()
    bits[0, 0] |= np.uint64(1) << np.uint64(50)  # chunk 50 >= n = 48
    assert _status(mpt, inst.weights, bits) == 1
    big = I.random_instance(33, 40, 3, seed=1)
    assert _status(mpt, big.weights, big.bits) == 2
    huge = I.Instance(np.full(4, 1 << 61, dtype=np.int64), I.pack_requests([[0, 1], [2, 3], [0]], 4))
    assert _status(mpt, huge.weights, huge.bits) == 3


def test_workspace_and_modes(mpt):
    inst = I.config(2)  # m = 20
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    auto = mpt.mpt_workspace_bytes(ctx)
    N = 1 << 20
    assert auto >= N * (8 + 8 + 4 + 4 + 4)  # wI, F, split and the two blocked tables
    mpt.mpt_set_dp_mode(ctx, "general")
    assert N * 20 <= mpt.mpt_workspace_bytes(ctx) < auto
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_layout(ctx)
    assert e.value.status == 7
    heavy = I.Instance(np.full(20, 60000, dtype=np.int64), inst.bits)  # sum_i w(R_i) >= 2^20
    ctx2 = mpt.mpt_create(heavy.weights, heavy.bits)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_dp_mode(ctx2, "blocked")
    assert e.value.status == 3
    # AUTO takes the 64-bit-key tiles there: uint64 working tables and per-block slots
    heavy_auto = mpt.mpt_workspace_bytes(ctx2)
    assert heavy_auto >= N * (8 + 8 + 4 + 8 + 8)
    mpt.mpt_set_dp_mode(ctx2, "wide")
    assert mpt.mpt_workspace_bytes(ctx2) == heavy_auto
    mpt.mpt_set_dp_mode(ctx, "wide")  # allowed for light weights too
    assert mpt.mpt_workspace_bytes(ctx) == heavy_auto
    huge = I.Instance(np.full(20, 1 << 47, dtype=np.int64), inst.bits)  # sum_i w(R_i) >= 2^51
    ctx3 = mpt.mpt_create(huge.weights, huge.bits)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_dp_mode(ctx3, "wide")
    assert e.value.status == 3
    mpt.mpt_set_dp_mode(ctx3, "auto")
    assert N * 20 <= mpt.mpt_workspace_bytes(ctx3) < auto  # the general kernels
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_dp_mode(ctx3, 4)
    assert e.value.status == 1
    mpt.mpt_destroy(ctx)
    mpt.mpt_destroy(ctx2)
    mpt.mpt_destroy(ctx3)


def test_status_strings(mpt):
    lib = mpt.load()
    for code in range(10):
        assert lib.mpt_status_string(code)


def _batch_status(mpt, weights, instances):
    try:
        b = mpt.mpt_batch_create(weights, *mpt.pack_batch(instances))
        mpt.mpt_batch_destroy(b)
        return 0
    except mpt.MPTError as e:
        return e.status


def test_batch_create_validation(mpt):
    w = np.ones(50, dtype=np.int64)
    assert _batch_status(mpt, w, [[[1, 2], [3]], [[4]]]) == 0
    assert _batch_status(mpt, w, [[[i] for i in range(14)]]) == 0           # m = 14
    assert _batch_status(mpt, w, [[[i] for i in range(16)]]) == 0           # m = 16 (packed keys)
    assert _batch_status(mpt, w, [[[i] for i in range(17)]]) == 2           # m > 16
    heavy16 = np.full(50, 1 << 12, dtype=np.int64)
    assert _batch_status(mpt, heavy16, [[[0, 1]] * 8 + [[2]] * 8]) == 2    # m = 16, shared weight >= 2^16
    assert _batch_status(mpt, w, [[[1, 1]]]) == 1                           # repeated chunk in a request
    assert _batch_status(mpt, w, [[[50]]]) == 1                             # chunk id >= n
    assert _batch_status(mpt, w, [[]]) == 1                                 # an instance with no request
    heavy = np.full(50, 1 << 30, dtype=np.int64)
    assert _batch_status(mpt, heavy, [[[0, 1], [0, 1], [2]]]) == 3          # shared weight >= 2^31
    assert _batch_status(mpt, heavy, [[[0, 1]], [[0, 3], [0, 4]]]) == 0     # private and common chunks only
    huge = np.full(50, 1 << 61, dtype=np.int64)
    assert _batch_status(mpt, huge, [[[0, 1], [0, 1]]]) == 3                # sum of w(R_i) >= 2^62
    big = [[list(range(0, 2049))]]
    assert _batch_status(mpt, np.ones(3000, dtype=np.int64), big) == 2      # > 2048 occurrences
    m14 = [[list(range(146 * i, 146 * i + 146)) for i in range(14)]]
    assert _batch_status(mpt, np.ones(3000, dtype=np.int64), m14) == 0      # m = 14, 2044 occurrences
    # m = 15 on 64-bit keys (the per-subset kernel): 1024 occurrences at most
    w200 = np.full(3000, 200, dtype=np.int64)
    m15 = [[list(range(35 * i, 35 * i + 70)) for i in range(15)]]
    assert _batch_status(mpt, w200, m15) == 2                               # 1050 occurrences
    m15 = [[list(range(34 * i, 34 * i + 68)) for i in range(15)]]
    assert _batch_status(mpt, w200, m15) == 0                               # 1020 occurrences
    # m = 15 on packed keys (the row-blocked kernel): up to 2048
    m15 = [[list(range(136 * i, 136 * i + 136)) for i in range(15)]]
    assert _batch_status(mpt, np.ones(3000, dtype=np.int64), m15) == 0      # 2040 occurrences


def test_schedule_and_cache_validation(mpt):
    """Argument checks of mpt_serve_order / mpt_cache_costs / mpt_layout_pinned
    happen on the host, before any CUDA call."""
    import ctypes

    lib = mpt.load()
    i64p, i32p = ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int32)

    def p64(a):
        return np.ascontiguousarray(a, dtype=np.int64).ctypes.data_as(i64p)

    w = np.ones(5, dtype=np.int64)
    offs = np.array([0, 2, 3], dtype=np.int64)
    ch = np.array([0, 1, 4], dtype=np.int64)
    out = np.zeros(2, dtype=np.int32)
    o32 = out.ctypes.data_as(i32p)

    def order_status(n, m, offs, ch, arrival=None, window=0):
        arr = None if arrival is None else np.ascontiguousarray(arrival, dtype=np.int32).ctypes.data_as(i32p)
        return lib.mpt_serve_order(n, m, p64(offs), p64(ch), arr, window, None, o32)

    assert order_status(5, 0, offs, ch) == 1                          # m < 1
    assert order_status(5, 2, np.array([1, 2, 3]), ch) == 1            # offsets not from 0
    assert order_status(5, 2, np.array([0, 3, 2]), ch) == 1            # decreasing offsets
    assert order_status(4, 2, offs, ch) == 1                          # chunk id >= n
    assert order_status(5, 2, offs, ch, arrival=[0, 0]) == 1          # arrival not a permutation
    assert order_status(5, 2, offs, ch, window=-1) == 1               # negative window
    long_offs = np.array([0, 4097], dtype=np.int64)
    assert order_status(5000, 1, long_offs, np.arange(4097)) == 2     # string longer than 4096

    caps = np.array([0, 3], dtype=np.int64)
    costs = np.zeros(2, dtype=np.int64)

    def cache_status(w, caps, n_caps, order=None):
        o = None if order is None else np.ascontiguousarray(order, dtype=np.int32).ctypes.data_as(i32p)
        return lib.mpt_cache_costs(p64(w), int(len(w)), 2, p64(offs), p64(ch), o, p64(caps), n_caps, None,
                                   costs.ctypes.data_as(i64p), None)

    assert cache_status(w, caps, -1) == 1                              # negative count
    assert cache_status(w, caps, 1025) == 1                            # more than 1024 capacities
    assert cache_status(w, np.array([-1, 3]), 2) == 1                  # negative capacity
    assert cache_status(np.array([1, 1, 0, 1, 1]), caps, 2) == 1       # weight 0
    assert cache_status(w, caps, 2, order=[1, 1]) == 1                 # order not a permutation
    big = np.full(5, 1 << 61, dtype=np.int64)
    assert cache_status(big, caps, 2) == 3                             # total weight >= 2^62

    perm = np.zeros(3, dtype=np.int64)

    def pinned_status(m, offs, ch, t, method):
        return lib.mpt_layout_pinned(p64(w), 5, m, p64(offs), p64(ch), t, method, None,
                                     perm.ctypes.data_as(i64p), None, None)

    assert pinned_status(2, offs, ch, -1, 0) == 1                      # t < 0
    assert pinned_status(2, offs, ch, 1, 7) == 1                       # unknown method
    assert pinned_status(2, offs, np.array([0, 1, 9]), 1, 0) == 1      # chunk id >= n
    assert pinned_status(2, offs, np.array([0, 0, 4]), 0, 0) == 1      # repeated chunk in a request
    o33 = np.arange(34, dtype=np.int64) % 3
    assert pinned_status(33, np.arange(34, dtype=np.int64), o33, 0, 0) == 2  # exact method beyond 32


def test_staged_solve_host_checks(mpt):
    """Step counts and the state checks of the staged solve need no GPU."""
    import ctypes

    lib = mpt.load()
    inst = I.random_instance(14, 40, 3, seed=2)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    n = ctypes.c_int32()
    assert lib.mpt_solve_steps(ctx.handle, ctypes.byref(n)) == 0 and n.value == 3  # tile layers 0..2
    mpt.mpt_set_dp_mode(ctx, "general")
    assert lib.mpt_solve_steps(ctx.handle, ctypes.byref(n)) == 0 and n.value == 14  # singletons + sizes 2..14
    opt = ctypes.c_int64()
    assert lib.mpt_solve_layers(ctx.handle, None, 0, None, 1, None) == 7  # nothing begun
    assert lib.mpt_solve_end(ctx.handle, None, 0, None, ctypes.byref(opt)) == 7
    fake = ctypes.c_void_p(1 << 20)
    assert lib.mpt_solve_resume(ctx.handle, fake, 1 << 30, 0) == 1  # step 0 is not resumable
    assert lib.mpt_solve_resume(ctx.handle, fake, 1 << 30, 15) == 1  # past the last step
    assert lib.mpt_solve_resume(ctx.handle, None, 1 << 30, 1) == 1  # needs a workspace
    mpt.mpt_destroy(ctx)


def test_lean_tables_host_checks(mpt):
    import ctypes

    lib = mpt.load()
    inst = I.random_instance(14, 40, 3, seed=2)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    full = mpt.mpt_workspace_bytes(ctx)
    assert lib.mpt_set_tables(ctx.handle, 2) == 1
    assert lib.mpt_set_tables(ctx.handle, 1) == 0
    lean = mpt.mpt_workspace_bytes(ctx)
    assert full - lean == 12 * (1 << 14)  # 16 bytes of w(I) and F become 4
    pF, pS, pW = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    assert lib.mpt_tables(ctx.handle, ctypes.byref(pF), ctypes.byref(pW), ctypes.byref(pS)) == 1  # lean: no int64 tables
    assert lib.mpt_tables32(ctx.handle, ctypes.byref(pF), ctypes.byref(pS)) == 7  # not solved yet
    assert lib.mpt_set_tables(ctx.handle, 0) == 0
    assert lib.mpt_tables32(ctx.handle, ctypes.byref(pF), ctypes.byref(pS)) == 1  # int64 layout
    mpt.mpt_destroy(ctx)
    heavy = I.random_instance(8, 16, 4, seed=3, wmin=1 << 27, wmax=1 << 28)  # sum_i w(R_i) >= 2^31
    ctx = mpt.mpt_create(heavy.weights, heavy.bits)
    assert lib.mpt_set_tables(ctx.handle, 1) == 3
    mpt.mpt_destroy(ctx)


def test_helper_argument_checks(mpt):
    """Host-side checks of mpt_trie_cost, mpt_solve_noalloc,
    mpt_gather_bandwidth and mpt_alu_addmin_peak, all returned before any CUDA
    call."""
    import ctypes

    lib = mpt.load()
    p64 = lambda a: a.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))
    w = np.array([3, 4, 5], dtype=np.int64)
    cost = ctypes.c_int64()
    offs = np.array([0, 2, 3], dtype=np.int64)
    ch = np.array([0, 1, 2], dtype=np.int64)
    assert lib.mpt_trie_cost(None, 3, 2, p64(offs), p64(ch), ctypes.byref(cost)) == 1
    assert lib.mpt_trie_cost(p64(w), 3, 0, p64(offs), p64(ch), ctypes.byref(cost)) == 1
    bad_first = np.array([1, 2, 3], dtype=np.int64)
    assert lib.mpt_trie_cost(p64(w), 3, 2, p64(bad_first), p64(ch), ctypes.byref(cost)) == 1
    decreasing = np.array([0, 2, 1], dtype=np.int64)
    assert lib.mpt_trie_cost(p64(w), 3, 2, p64(decreasing), p64(ch), ctypes.byref(cost)) == 1
    out_of_range = np.array([0, 1, 3], dtype=np.int64)
    assert lib.mpt_trie_cost(p64(w), 3, 2, p64(offs), p64(out_of_range), ctypes.byref(cost)) == 1
    zero_w = np.array([3, 0, 5], dtype=np.int64)
    assert lib.mpt_trie_cost(p64(zero_w), 3, 2, p64(offs), p64(ch), ctypes.byref(cost)) == 1
    # mpt_solve_noalloc: null device pointers, then m beyond its 20-request limit
    dummy = ctypes.c_void_p(256)
    args = [dummy, 3, dummy, 21, dummy, dummy, dummy, dummy, None]
    assert lib.mpt_solve_noalloc(None, *args[1:]) == 1
    assert lib.mpt_solve_noalloc(*args) == 2
    assert lib.mpt_solve_noalloc(dummy, 0, dummy, 5, dummy, dummy, dummy, dummy, None) == 1
    # mpt_gather_bandwidth: table size and load count
    gbps = ctypes.c_double()
    assert lib.mpt_gather_bandwidth(9, 1000, None, ctypes.byref(gbps)) == 1
    assert lib.mpt_gather_bandwidth(33, 1000, None, ctypes.byref(gbps)) == 1
    assert lib.mpt_gather_bandwidth(20, 0, None, ctypes.byref(gbps)) == 1
    assert lib.mpt_gather_bandwidth(20, 1000, None, None) == 1
    # mpt_alu_addmin_peak: operation count and output
    rate = ctypes.c_double()
    assert lib.mpt_alu_addmin_peak(0, None, ctypes.byref(rate)) == 1
    assert lib.mpt_alu_addmin_peak(1000, None, None) == 1


def test_caller_workspace_checks(mpt):
    """A caller workspace below mpt_workspace_bytes() or off a 256-byte
    boundary is refused by mpt_solve, mpt_solve_begin and mpt_solve_resume
    before any copy or launch (the fake pointers are never dereferenced)."""
    import ctypes

    lib = mpt.load()
    inst = I.random_instance(12, 30, 3, seed=4)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    need = mpt.mpt_workspace_bytes(ctx)
    opt = ctypes.c_int64()
    aligned, misaligned = ctypes.c_void_p(1 << 20), ctypes.c_void_p((1 << 20) + 16)
    assert lib.mpt_solve(ctx.handle, aligned, need - 1, None, ctypes.byref(opt)) == 5
    assert lib.mpt_solve(ctx.handle, misaligned, need, None, ctypes.byref(opt)) == 1
    assert lib.mpt_solve(ctx.handle, aligned, need, None, None) == 1  # no place for OPT
    assert lib.mpt_solve(None, aligned, need, None, ctypes.byref(opt)) == 1
    assert lib.mpt_solve_begin(ctx.handle, aligned, need - 256, None) == 5
    assert lib.mpt_solve_begin(ctx.handle, misaligned, need, None) == 1
    assert lib.mpt_solve_resume(ctx.handle, aligned, need - 1, 1) == 5
    assert lib.mpt_solve_resume(ctx.handle, misaligned, need, 1) == 1
    # a refused call leaves nothing begun and nothing solved
    assert lib.mpt_solve_layers(ctx.handle, aligned, need, None, 1, None) == 7
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_layout(ctx)
    assert e.value.status == 7
    mpt.mpt_destroy(ctx)


def test_key_width_follows_shared_weight(mpt):
    """The packed-key limits apply to the shared weight: private suffixes and
    a common prefix of 2^40 tokens keep the 32-bit keys (BLOCKED accepted,
    the narrow workspace); a chunk of 2^20 tokens that some but not all
    requests share does not."""
    base = I.config(1)  # m = 12
    heavy_private = I.with_query_chunks(base, 1 << 40, 1 << 40, seed=1)
    narrow = mpt.mpt_create(base.weights, base.bits)
    ctx = mpt.mpt_create(heavy_private.weights, heavy_private.bits)
    assert mpt.mpt_workspace_bytes(ctx) - mpt.mpt_workspace_bytes(narrow) < 4096  # the inputs grow by 12 chunks
    mpt.mpt_set_dp_mode(ctx, "blocked")
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_tables(ctx, "lean")  # the int32 tables still need sum_i w(R_i) < 2^31
    assert e.value.status == 3
    prefix = I.with_common_prefix(heavy_private, 1 << 40)  # plus 2^40 tokens in every request
    ctx_p = mpt.mpt_create(prefix.weights, prefix.bits)
    mpt.mpt_set_dp_mode(ctx_p, "blocked")
    mpt.mpt_destroy(ctx_p)
    shared = I.Instance(base.weights.copy(), base.bits)
    x = int(np.flatnonzero(np.unpackbits(base.bits[0].view(np.uint8), bitorder="little"))[0])
    assert W.request_counts(base)[x] >= 2
    shared.weights[x] = 1 << 20  # a chunk of request 0 that other requests hold too
    ctx2 = mpt.mpt_create(shared.weights, shared.bits)
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_set_dp_mode(ctx2, "blocked")
    assert e.value.status == 3
    for c in (narrow, ctx, ctx2):
        mpt.mpt_destroy(c)


def test_blocked_limit_on_shared_weight_property(mpt):
    """Host logic of the key-width choice on random instances: BLOCKED is
    accepted exactly when the shared weight (sum_i w(R_i) less the chunks
    one request alone or all m >= 2 requests hold) is below 2^(32 - b),
    b = min(m, 12) tile bits (2^20 from m = 12 on), and WIDE exactly when it
    is below 2^51."""
    rng = np.random.default_rng(404)
    for t in range(60):
        m = int(rng.integers(1, 15))
        n = int(rng.integers(1, 40))
        base = I.random_instance(m, n, (0, n), seed=int(rng.integers(1 << 30)), wmin=1, wmax=9, allow_empty=True)
        if t % 3 == 0:
            base = I.with_common_prefix(base, int(rng.integers(1, 1 << 40)))
        shared = W.shared_weight(base)
        for limit, mode in ((1 << (32 - min(m, 12)), "blocked"), (1 << 51, "wide")):
            # scale so that the shared weight lands just below or at the limit when it is positive
            for target in (limit - 1, limit):
                scale = max(1, target // shared) if shared > 0 else 1
                if max(int(x) for x in base.weights) * scale * max(m, 1) >= 1 << 62:
                    continue  # beyond the int64 sums the ABI accepts
                inst = I.Instance(base.weights * scale, base.bits)
                if W.request_weight_sum(inst) >= 1 << 62:
                    continue
                ctx = mpt.mpt_create(inst.weights, inst.bits)
                ok = W.shared_weight(inst) < limit
                try:
                    mpt.mpt_set_dp_mode(ctx, mode)
                    accepted = True
                except mpt.MPTError as e:
                    assert e.status == 3
                    accepted = False
                assert accepted == ok, (t, mode, W.shared_weight(inst))
                mpt.mpt_destroy(ctx)


def test_binding_fails_loudly_without_the_library(tmp_path):
    """No fallback: with the CUDA library absent, the binding refuses to load
    instead of computing anything elsewhere."""
    import subprocess
    import sys

    code = (
        "import pathlib, sys\n"
        "from paper_2609_13692_gb300 import build as B, mpt\n"
        f"B.LIB = pathlib.Path({str(tmp_path / 'absent' / 'libmpt.so')!r})\n"
        "mpt._LIB = None\n"
        "try:\n"
        "    mpt.solve([3, 4], [[1], [3]])\n"
        "except RuntimeError as e:\n"
        "    print('refused:', e)\n"
        "    sys.exit(0)\n"
        "sys.exit(1)\n"
    )
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "is missing" in r.stdout


def test_device_allocation_failure(mpt, monkeypatch):
    """With MPT_FAIL_DEVICE_ALLOC=1 every allocation the library makes for
    itself fails as an exhausted device would: each entry point returns
    MPT_ERR_OUT_OF_MEMORY before any CUDA call and writes no output, and the
    context stays unsolved (no GPU needed)."""
    import ctypes

    lib = mpt.load()
    inst = I.config(1)
    ctx = mpt.mpt_create(inst.weights, inst.bits)
    monkeypatch.setenv("MPT_FAIL_DEVICE_ALLOC", "1")
    opt = ctypes.c_int64(-7)
    assert lib.mpt_solve(ctx.handle, None, 0, None, ctypes.byref(opt)) == 4
    assert opt.value == -7
    offs = np.full(inst.m + 1, -7, dtype=np.int64)
    chunks = np.full(64, -7, dtype=np.int64)
    dfs = np.full(inst.m, -7, dtype=np.int32)
    assert lib.mpt_layout(ctx.handle, offs.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                          chunks.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                          dfs.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))) == 7
    assert (offs == -7).all() and (chunks == -7).all() and (dfs == -7).all()
    assert lib.mpt_solve_begin(ctx.handle, None, 0, None) == 4
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_trie_cost(inst.weights, np.array([0, 1, 2], dtype=np.int64), np.array([0, 1], dtype=np.int64))
    assert e.value.status == 4
    reqs = [[0, 1, 2], [1, 2, 3], [2, 3, 4]]
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_greedy(np.arange(1, 6, dtype=np.int64), reqs)
    assert e.value.status == 4
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_serve_order(5, reqs)
    assert e.value.status == 4
    with pytest.raises(mpt.MPTError) as e:
        mpt.mpt_cache_costs(np.arange(1, 6, dtype=np.int64), reqs, [3, 10])
    assert e.value.status == 4
    b = mpt.mpt_batch_create(np.arange(1, 6, dtype=np.int64), *mpt.pack_batch([reqs, reqs[:2]]))
    assert lib.mpt_batch_solve(b.handle, None, 0, None) == 4
    monkeypatch.delenv("MPT_FAIL_DEVICE_ALLOC")

"""Batched small-instance solver (mpt_batch_*) against the oracle, per instance.

Every instance of a batch must match the oracle bit for bit: OPT, every F(S)
and split(S) of its own 2^m table, every request's chunk order and the DFS
order.  The batches mix sizes m = 1..16, empty and repeated requests, and
RAG-like groups drawn from topical pools (the shape of the paper's request
groups, Sec. 7).
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


def rag_batch(count, n, seed, m_range=(1, 13), k_range=(0, 10), pool_size=40):
    rng = np.random.default_rng(seed)
    weights = rng.integers(1, 501, size=n, dtype=np.int64)
    pools = [rng.choice(n, size=pool_size, replace=False) for _ in range(16)]
    batch = []
    for _ in range(count):
        m = int(rng.integers(m_range[0], m_range[1] + 1))
        pool = pools[int(rng.integers(len(pools)))]
        reqs = []
        for _ in range(m):
            k = int(rng.integers(k_range[0], k_range[1] + 1))
            src = pool if rng.random() < 0.8 else np.arange(n)
            reqs.append(sorted(set(int(x) for x in rng.choice(src, size=k, replace=False))))
        batch.append(reqs)
    return weights, batch


def check_batch(mpt, weights, batch):
    opt, perms, orders, b = mpt.solve_batch(weights, batch)
    F_all, S_all, offs = mpt.mpt_batch_tables(b)
    F_all = F_all.cpu().numpy()
    S_all = S_all.cpu().numpy().view(np.uint32)
    n = int(weights.shape[0])
    for i, reqs in enumerate(batch):
        bits = I.pack_requests(reqs, n)
        o_opt, oF, owI, osplit = O.solve(weights, bits)
        assert opt[i] == o_opt, (i, opt[i], o_opt)
        lo, hi = int(offs[i]), int(offs[i + 1])
        assert np.array_equal(F_all[lo:hi], oF), i
        assert np.array_equal(S_all[lo:hi], osplit), i
        o_perms, o_dfs = O.layout(weights, bits, osplit)
        assert perms[i] == o_perms, i
        assert orders[i] == o_dfs, i


def test_batch_rag_groups(mpt):
    weights, batch = rag_batch(300, 3000, seed=1)
    check_batch(mpt, weights, batch)


def test_batch_edge_cases(mpt):
    w = np.arange(1, 21, dtype=np.int64)
    batch = [
        [[3]],                                   # m = 1
        [[], [1, 2], []],                        # empty requests
        [[1, 2, 3]] * 13,                        # identical requests, m = 13
        [[i] for i in range(13)],                # disjoint singletons
        [[x for x in range(13) if x != i] for i in range(13)],  # leave-one-out L_13
        [[0, 19], [19], [0]],
    ]
    check_batch(mpt, w, batch)
    opt, perms, orders, b = mpt.solve_batch(np.ones(13, dtype=np.int64),
                                            [[[x for x in range(13) if x != i] for i in range(13)]])
    assert opt[0] == O.loo_free(13)


def test_batch_large_requests(mpt):
    """Requests of up to 150 chunks (near the 2048-occurrence limit at m = 13)."""
    weights, batch = rag_batch(40, 20000, seed=2, m_range=(10, 13), k_range=(100, 150), pool_size=400)
    check_batch(mpt, weights, batch)


def test_batch_fourteen_and_fifteen_requests(mpt):
    """Groups of 14 and 15 requests: RAG-shaped groups on the packed keys
    (row-blocked kernel, split table in global memory, phase A in passes),
    heavy groups on the 64-bit keys (per-subset kernel), groups with private
    suffixes and a common prefix, and a 15-request group at the
    1024-occurrence limit, mixed with smaller sizes."""
    weights, batch = rag_batch(24, 3000, seed=14, m_range=(14, 15), k_range=(0, 10))
    rng = np.random.default_rng(15)
    n = int(weights.shape[0])
    heavy_ids = n
    weights = np.concatenate([weights, rng.integers(1 << 18, 1 << 20, size=40, dtype=np.int64)])
    for _ in range(4):
        m = int(rng.integers(14, 16))
        batch.append([sorted(set(int(x) for x in heavy_ids + rng.choice(40, size=int(rng.integers(1, 8)),
                                                                        replace=False))) for _ in range(m)])
    prefix = len(weights)
    weights = np.concatenate([weights, [1 << 35], rng.integers(1 << 30, 1 << 40, size=15, dtype=np.int64)])
    grp = [sorted(set(int(x) for x in rng.choice(300, size=6, replace=False))) + [prefix, prefix + 1 + i]
           for i in range(15)]
    batch.append(grp)
    batch.append([list(range(68 * i, 68 * i + 68)) for i in range(15)])
    batch += rag_batch(20, 3000, seed=16, m_range=(1, 13))[1]
    shared = [_shared_weight(weights, reqs) for reqs in batch if len(reqs) >= 14]
    assert any(s >= 1 << 17 for s in shared) and any(s < 1 << 17 for s in shared)
    check_batch(mpt, weights, batch)


def test_batch_sixteen_requests(mpt):
    """Groups of 16 requests (packed keys only; the row-blocked kernel with
    its rows in a global scratch slot per block), RAG-shaped with light
    passages, one with private suffixes and a common prefix, and the
    leave-one-out family L_16 (its optimum has a closed form), mixed with
    smaller sizes."""
    weights, batch = rag_batch(12, 3000, seed=161, m_range=(16, 16), k_range=(0, 8))
    weights = (weights % 97) + 1
    rng = np.random.default_rng(162)
    prefix = len(weights)
    weights = np.concatenate([weights, [1 << 33], rng.integers(1 << 30, 1 << 38, size=16, dtype=np.int64)])
    batch.append([sorted(set(int(x) for x in rng.choice(300, size=5, replace=False))) + [prefix, prefix + 1 + i]
                  for i in range(16)])
    batch.append([[x for x in range(16) if x != i] for i in range(16)])
    batch += rag_batch(10, 3000, seed=163, m_range=(12, 15))[1]
    assert all(_shared_weight(weights, reqs) < 1 << 16 for reqs in batch if len(reqs) == 16)
    check_batch(mpt, weights, batch)


def _shared_weight(weights, reqs):
    """sum_i w(R_i) less the chunks that one or all m >= 2 requests hold."""
    cnt = {}
    for r in reqs:
        for x in r:
            cnt[x] = cnt.get(x, 0) + 1
    return sum(int(weights[x]) * c for x, c in cnt.items() if 2 <= c < len(reqs))


def test_batch_mixed_key_widths(mpt):
    """Instances whose shared weight needs the 64-bit keys (>= 2^(32 - m))
    next to ones that use the packed 32-bit keys, sizes shuffled so the
    per-size launches must map results back to their instances."""
    rng = np.random.default_rng(71)
    n = 400
    heavy = rng.integers(60_000, 120_000, size=n, dtype=np.int64)
    batch = []
    for _ in range(60):
        m = int(rng.integers(2, 14))
        pool = rng.choice(n, size=30, replace=False)
        batch.append([sorted(set(int(x) for x in rng.choice(pool, size=int(rng.integers(1, 12)), replace=False)))
                      for _ in range(m)])
    shared = [_shared_weight(heavy, reqs) for reqs in batch]
    assert any(s >= 1 << (32 - len(reqs)) for s, reqs in zip(shared, batch))
    assert any(s < 1 << (32 - len(reqs)) for s, reqs in zip(shared, batch))
    check_batch(mpt, heavy, batch)


def test_batch_private_and_common_weights(mpt):
    """Groups whose requests carry a private suffix of up to 2^40 tokens and a
    common prefix of up to 2^36 (sum_i w(R_i) far beyond 2^31) over small
    shared passages: the shared weight keeps them on the 32-bit keys, and
    every OPT, table entry and order equals the oracle's."""
    weights, batch = rag_batch(200, 3000, seed=5, m_range=(1, 13))
    rng = np.random.default_rng(6)
    extra = []
    for g, reqs in enumerate(batch):
        prefix = len(weights) + len(extra)
        extra.append(int(rng.integers(1 << 30, 1 << 36)))
        for i in range(len(reqs)):
            if rng.random() < 0.7:
                reqs[i] = reqs[i] + [len(weights) + len(extra)]
                extra.append(int(rng.integers(1 << 20, 1 << 40)))
            if g % 2 == 0:
                reqs[i] = [prefix] + reqs[i]
    w = np.concatenate([weights, np.array(extra, dtype=np.int64)])
    assert all(_shared_weight(w, reqs) < 1 << (32 - len(reqs)) for reqs in batch)
    assert max(sum(int(w[x]) for r in reqs for x in r) for reqs in batch) >= 1 << 40
    check_batch(mpt, w, batch)

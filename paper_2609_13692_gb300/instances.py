"""Seeded synthetic instances of the Minimum-Prefix-Trie problem (Sec. 2).

An instance is a chunk universe ``U = {0, .., n-1}`` with positive integer
token weights ``w`` and ``m`` requests ``R_i ⊆ U`` (Sec. 2, eq. 1).  It is
stored as two arrays:

* ``weights``: ``int64[n]``, ``weights[x] = w(x) >= 1``;
* ``bits``: ``uint64[m, ceil(n / 64)]``, row-major; bit ``x % 64`` of word
  ``x // 64`` in row ``i`` is set iff chunk ``x`` belongs to request ``R_i``.

This module only draws random numbers and packs bits.  It holds none of the
solver's arithmetic, so both the CUDA path and the CPU oracle can be fed from
it without sharing any of the method.

The workloads follow the shapes the paper describes: Zipf-distributed
retrieval over topical pools (Sec. 6.2, Sec. 7), the leave-one-out family
``L_n`` (Sec. 5) and the paper's small worked examples (Thm 4, Sec. 6.3,
Sec. 10.1).  The paper's own BEIR traces are not available, so the RAG-shaped
generators stand in for them with the statistics the paper reports (k = 5..40
passages per request, most passages shared by a few requests).
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

__all__ = [
    "Instance",
    "pack_requests",
    "unpack_requests",
    "zipf_small",
    "leave_one_out",
    "rag_pools",
    "rag_ranked",
    "stream",
    "STREAMS",
    "config",
    "CONFIGS",
    "random_instance",
    "with_query_chunks",
    "with_common_prefix",
    "k4_3",
    "open_problem_k4",
    "tightness_witness",
]


@dataclass
class Instance:
    """A packed MPT instance plus a short description of how it was drawn."""

    weights: np.ndarray  # int64[n]
    bits: np.ndarray  # uint64[m, ceil(n/64)]
    name: str = ""

    @property
    def m(self) -> int:
        return int(self.bits.shape[0])

    @property
    def n(self) -> int:
        return int(self.weights.shape[0])

    def requests(self) -> list[list[int]]:
        return unpack_requests(self.bits, self.n)


def pack_requests(requests, n: int) -> np.ndarray:
    """Pack a list of chunk-id collections into the ``uint64[m, ceil(n/64)]`` layout."""
    m = len(requests)
    words = max(1, (n + 63) // 64)
    bits = np.zeros((m, words), dtype=np.uint64)
    for i, req in enumerate(requests):
        ids = np.asarray(sorted(set(int(x) for x in req)), dtype=np.int64)
        if ids.size == 0:
            continue
        if ids.min() < 0 or ids.max() >= n:
            raise ValueError(f"request {i} has a chunk id outside [0, {n})")
        np.bitwise_or.at(bits[i], ids >> 6, np.left_shift(np.uint64(1), (ids & 63).astype(np.uint64)))
    return bits


def unpack_requests(bits: np.ndarray, n: int) -> list[list[int]]:
    """Inverse of :func:`pack_requests`: sorted chunk ids per request."""
    out = []
    for row in np.asarray(bits, dtype=np.uint64):
        as_bytes = row.astype("<u8").view(np.uint8)
        flags = np.unpackbits(as_bytes, bitorder="little")[:n]
        out.append(np.flatnonzero(flags).tolist())
    return out


def _finite_zipf_cdf(count: int, s: float) -> np.ndarray:
    ranks = np.arange(1, count + 1, dtype=np.float64)
    p = ranks ** (-s)
    cdf = np.cumsum(p)
    return cdf / cdf[-1]


def _draw_distinct(rng: np.random.Generator, k: int, draw_one) -> list[int]:
    chosen: list[int] = []
    seen: set[int] = set()
    while len(chosen) < k:
        x = int(draw_one())
        if x in seen:
            continue  # redraw duplicates
        seen.add(x)
        chosen.append(x)
    return chosen


def zipf_small(m: int = 12, n: int = 48, k: int = 5, s: float = 1.0, wmin: int = 64, wmax: int = 512,
               seed: int = 0) -> Instance:
    """Each request draws ``k`` distinct ids by finite Zipf(s) over ``n`` ids
    (P(id = j) proportional to (j+1)^-s); weights uniform integers in [wmin, wmax]."""
    rng = np.random.default_rng(seed)
    cdf = _finite_zipf_cdf(n, s)
    weights = rng.integers(wmin, wmax + 1, size=n, dtype=np.int64)
    reqs = []
    for _ in range(m):
        reqs.append(_draw_distinct(rng, k, lambda: min(int(np.searchsorted(cdf, rng.random(), side="right")), n - 1)))
    return Instance(weights, pack_requests(reqs, n), f"zipf m={m} n={n} k={k} s={s} seed={seed}")


def leave_one_out(n: int) -> Instance:
    """The leave-one-out family L_n (Sec. 5): U = [n], R_i = U \\ {i}, unit weights."""
    weights = np.ones(n, dtype=np.int64)
    reqs = [[x for x in range(n) if x != i] for i in range(n)]
    return Instance(weights, pack_requests(reqs, n), f"leave-one-out n={n}")


def _rag_draw(m: int, n: int, pools: int, pool_size: int, k: int, tail_s: float, seed: int, p_pool: float,
              w_mean: float, w_sigma: float, wmin: int, wmax: int):
    """Weights and per-request passage lists, in draw order (see rag_pools)."""
    rng = np.random.default_rng(seed)
    mu = math.log(w_mean) - w_sigma * w_sigma / 2.0
    weights = np.clip(np.rint(rng.lognormal(mu, w_sigma, size=n)), wmin, wmax).astype(np.int64)
    pool_ids = rng.choice(n, size=pools * pool_size, replace=False).reshape(pools, pool_size)
    tail_perm = rng.permutation(n)
    cdf = _finite_zipf_cdf(n, tail_s)

    def draw_tail() -> int:
        r = min(int(np.searchsorted(cdf, rng.random(), side="right")), n - 1)
        return int(tail_perm[r])

    reqs = []
    for _ in range(m):
        p = int(rng.integers(pools))

        def draw_one(p=p) -> int:
            if rng.random() < p_pool:
                return int(pool_ids[p, int(rng.integers(pool_size))])
            return draw_tail()

        reqs.append(_draw_distinct(rng, k, draw_one))
    return weights, reqs


def rag_pools(m: int, n: int, pools: int, pool_size: int, k: int, tail_s: float, seed: int = 0,
              p_pool: float = 0.8, w_mean: float = 150.0, w_sigma: float = 0.6, wmin: int = 32,
              wmax: int = 512) -> Instance:
    """RAG-shaped retrieval groups.

    The corpus has ``n`` passages.  ``pools`` disjoint topical pools of
    ``pool_size`` passages are drawn from it; a global tail ranks every passage
    (random permutation) under finite Zipf(``tail_s``).  Request i picks a pool
    uniformly; each of its ``k`` slots comes from that pool (uniformly) with
    probability ``p_pool``, else from the tail; duplicates are redrawn.
    Passage weights are lognormal with mean ``w_mean`` (mu = ln(mean) - sigma^2/2),
    rounded and clipped to [wmin, wmax].
    """
    weights, reqs = _rag_draw(m, n, pools, pool_size, k, tail_s, seed, p_pool, w_mean, w_sigma, wmin, wmax)
    return Instance(weights, pack_requests(reqs, n),
                    f"rag m={m} n={n} pools={pools}x{pool_size} k={k} tail_s={tail_s} seed={seed}")


def rag_ranked(m: int, n: int, pools: int, pool_size: int, k: int, tail_s: float, seed: int = 0,
               p_pool: float = 0.8, w_mean: float = 150.0, w_sigma: float = 0.6, wmin: int = 32,
               wmax: int = 512):
    """The requests of rag_pools as relevance-ranked lists (rank = draw order),
    in arrival order: (weights int64[n], list of m chunk-id lists)."""
    return _rag_draw(m, n, pools, pool_size, k, tail_s, seed, p_pool, w_mean, w_sigma, wmin, wmax)


# Request streams of the finite-cache study (Sec. 8): NFCorpus- and
# SciFact-shaped (k = 8 passages per query; about 6,000 tokens per request,
# i.e. passages of about 750 tokens), in arrival order.
STREAMS = {
    "nfcorpus-shaped": dict(m=2921, n=3633, pools=64, pool_size=40, k=8, tail_s=1.0, w_mean=750.0, wmin=64,
                            wmax=4096),
    "scifact-shaped": dict(m=1109, n=5183, pools=32, pool_size=60, k=8, tail_s=1.0, w_mean=750.0, wmin=64,
                           wmax=4096),
}


def stream(name: str, seed: int = 0):
    """(weights, ranked requests in arrival order) of a Sec. 8 stream."""
    c = dict(STREAMS[name])
    return rag_ranked(c.pop("m"), c.pop("n"), c.pop("pools"), c.pop("pool_size"), c.pop("k"), c.pop("tail_s"),
                      seed=seed, **c)


# The five workloads of the exact-solver benchmark, indexed 1..5.
CONFIGS = {
    1: dict(kind="zipf", m=12, n=48, k=5, s=1.0),
    2: dict(kind="loo", m=20, n=20),
    3: dict(kind="rag", m=24, n=100_000, pools=8, pool_size=200, k=10, tail_s=1.1),
    4: dict(kind="rag", m=28, n=100_000, pools=16, pool_size=300, k=20, tail_s=1.1),
    5: dict(kind="rag", m=30, n=1_000_000, pools=32, pool_size=400, k=40, tail_s=1.2),
    6: dict(kind="rag", m=31, n=100_000, pools=16, pool_size=300, k=20, tail_s=1.1),
    7: dict(kind="rag", m=32, n=100_000, pools=16, pool_size=300, k=20, tail_s=1.1),
}

CONFIG_NAMES = {
    1: "zipf-m12-n48-k5",
    2: "leave-one-out-n20",
    3: "rag-m24-n100k-8x200-k10",
    4: "rag-m28-n100k-16x300-k20",
    5: "rag-m30-n1M-32x400-k40",
    6: "rag-m31-n100k-16x300-k20",
    7: "rag-m32-n100k-16x300-k20",
}


def config(idx: int, seed: int = 0) -> Instance:
    """Workload ``idx`` (1..7) with the given seed (6, 7: the m = 31, 32 extensions)."""
    c = CONFIGS[idx]
    if c["kind"] == "zipf":
        inst = zipf_small(c["m"], c["n"], c["k"], c["s"], seed=seed)
    elif c["kind"] == "loo":
        inst = leave_one_out(c["n"])
    else:
        inst = rag_pools(c["m"], c["n"], c["pools"], c["pool_size"], c["k"], c["tail_s"], seed=seed)
    inst.name = f"{CONFIG_NAMES[idx]} ({inst.name})"
    return inst


def random_instance(m: int, n: int, k: int | tuple[int, int], seed: int, wmin: int = 1, wmax: int = 9,
                    allow_empty: bool = False) -> Instance:
    """Uniformly random requests of size k (or uniform in [k0, k1]) over n chunks."""
    rng = np.random.default_rng(seed)
    weights = rng.integers(wmin, wmax + 1, size=n, dtype=np.int64)
    reqs = []
    for _ in range(m):
        if isinstance(k, tuple):
            kk = int(rng.integers(k[0], k[1] + 1))
        else:
            kk = int(k)
        kk = min(kk, n)
        if kk == 0 and not allow_empty:
            kk = 1
        reqs.append(rng.choice(n, size=kk, replace=False).tolist())
    return Instance(weights, pack_requests(reqs, n), f"random m={m} n={n} k={k} seed={seed}")


def with_query_chunks(inst: Instance, wmin: int, wmax: int, seed: int, every: int = 1) -> Instance:
    """``inst`` with one new chunk appended to every ``every``-th request: a
    per-request suffix (its own question or document) that no other request
    holds, of weight uniform in [wmin, wmax]."""
    rng = np.random.default_rng(seed)
    reqs = inst.requests()
    owners = list(range(0, inst.m, every))
    extra = rng.integers(wmin, wmax + 1, size=len(owners), dtype=np.int64)
    n = inst.n + len(owners)
    for j, i in enumerate(owners):
        reqs[i] = list(reqs[i]) + [inst.n + j]
    weights = np.concatenate([inst.weights, extra])
    return Instance(weights, pack_requests(reqs, n), f"{inst.name} + query chunks [{wmin}, {wmax}]")


def with_common_prefix(inst: Instance, weight: int) -> Instance:
    """``inst`` with one new chunk of the given weight in every request: a
    system prompt or tool catalogue that all requests share."""
    reqs = [list(r) + [inst.n] for r in inst.requests()]
    weights = np.concatenate([inst.weights, np.array([weight], dtype=np.int64)])
    return Instance(weights, pack_requests(reqs, inst.n + 1), f"{inst.name} + common prefix {weight}")


def k4_3() -> Instance:
    """All four 3-subsets of {a,b,c,d} with unit weights (Thm 4)."""
    reqs = [[0, 1, 2], [0, 1, 3], [0, 2, 3], [1, 2, 3]]
    return Instance(np.ones(4, dtype=np.int64), pack_requests(reqs, 4), "K4^(3)")


def open_problem_k4() -> Instance:
    """The k = 4 instance on 7 chunks quoted under open problem 1 (Sec. 10.1), unit weights."""
    reqs = [[0, 1, 4, 5], [0, 2, 3, 6], [1, 2, 3, 6], [1, 2, 4, 5],
            [1, 3, 4, 5], [1, 4, 5, 6], [2, 3, 4, 6], [2, 3, 5, 6]]
    return Instance(np.ones(7, dtype=np.int64), pack_requests(reqs, 7), "open-problem-1 k=4")


def tightness_witness() -> Instance:
    """The four-request witness of Sec. 6.3: {0123},{14},{2578},{46}, unit weights."""
    reqs = [[0, 1, 2, 3], [1, 4], [2, 5, 7, 8], [4, 6]]
    return Instance(np.ones(9, dtype=np.int64), pack_requests(reqs, 9), "tightness witness")

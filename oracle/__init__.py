"""CPU oracle for the exact Minimum-Prefix-Trie solver.

TEST INFRASTRUCTURE ONLY: the plain, slow definition that the CUDA path is
checked against.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s ``cpu_baseline`` / ``--impl reference`` legs may import it.
It shares no code with the CUDA library and never imports it.

Everything here follows "Prefix Sharing Is a Sorting Problem" (arxiv
2609.13692):

* ``intersection_weights`` / ``dp`` / ``recompute`` / ``dp_at``: the C half
  (``oracle.c``): w(I(S)) by direct intersection (Thm 1 proof) and the
  O(3^m) subset recurrence of Sec. 3.1 in cost form (``dp_at``: its step at
  listed subsets, for timing samples of layers too large to finish).
* ``layout``: the constructive direction of Thm 1 -- walk the hierarchy
  top-down, at node B emit I(B) minus I(parent(B)), then recurse.
* ``trie_cost``: eq. (1), the weight of the non-root nodes of the trie of the
  laid-out strings, by building the trie.
* ``brute_force_permutations``: eq. (1) minimised over every choice of
  per-request permutations (OPT_free by definition, Sec. 2).
* ``brute_force_hierarchies``: eq. (2), min over all binary hierarchies of
  sum_x w(x) t_x(H), t_x counted as maximal clusters inside S_x (Sec. 3).
* ``brute_force_global_order``: OPT_glob, all pi_i induced by one chunk order.
* ``min_vertex_cover``: brute force tau(G) for Prop 2.
* ``spanning_tree_bound``: the lower bound of Sec. 6.3.
* ``radix_cache_cost``: a radix cache with LRU leaf eviction (Sec. 8, Thm 7).
* ``loo_free`` / ``loo_glob``: the closed forms of Thm 5.
* ``greedy``: the agglomerative common-intersection hierarchy of Sec. 6.2
  (Thm 6's H_g), with its layout and savings.
* ``trie_cost_sorted``: eq. (1) for many strings via lexicographic sorting.
* ``serve_order``: Thm 7's serving order (lexicographic order of the laid-out
  strings), optionally inside consecutive windows of arrivals (Sec. 8.1).
* ``radix_cache_costs``: ``radix_cache_cost`` over a list of capacities.
* ``pinned_layout`` / ``brute_force_pinned``: the Sec. 7.1 variant that pins
  each request's top-t passages, in relevance order, at the end.

Readings where the paper is silent are stated in ``oracle.c``'s header.
"""

from __future__ import annotations

import ctypes
import itertools
import math
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_BUILD = _HERE / "_build"
_LIB = None


def build(force: bool = False) -> Path:
    """Compile ``oracle.c`` into ``oracle/_build/liboracle.so`` with gcc."""
    _BUILD.mkdir(exist_ok=True)
    out = _BUILD / "liboracle.so"
    src = _HERE / "oracle.c"
    if force or not out.exists() or out.stat().st_mtime < src.stat().st_mtime:
        tmp = _BUILD / f"liboracle.{os.getpid()}.so"
        subprocess.run(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=c11", str(src), "-o", str(tmp)],
                       check=True)
        os.replace(tmp, out)
    return out


def _bind(lib):
    i64p = ctypes.POINTER(ctypes.c_int64)
    u64p = ctypes.POINTER(ctypes.c_uint64)
    u32p = ctypes.POINTER(ctypes.c_uint32)
    lib.oracle_wI_one.restype = ctypes.c_int64
    lib.oracle_wI_one.argtypes = [ctypes.c_int32, ctypes.c_int64, i64p, u64p, ctypes.c_uint64]
    lib.oracle_intersection_weights.restype = ctypes.c_int
    lib.oracle_intersection_weights.argtypes = [ctypes.c_int32, ctypes.c_int64, i64p, u64p, i64p]
    lib.oracle_dp.restype = ctypes.c_int
    lib.oracle_dp.argtypes = [ctypes.c_int32, i64p, i64p, u32p, ctypes.c_int32]
    lib.oracle_recompute.restype = ctypes.c_int
    lib.oracle_recompute.argtypes = [ctypes.c_int32, ctypes.c_int64, i64p, u64p, i64p, u64p, ctypes.c_int64,
                                     i64p, u32p, i64p, ctypes.c_int32]
    lib.oracle_dp_at.restype = ctypes.c_int
    lib.oracle_dp_at.argtypes = [ctypes.c_int32, i64p, i64p, u64p, ctypes.c_int64, i64p, u32p, ctypes.c_int32]
    lib.oracle_max_threads.restype = ctypes.c_int
    lib.oracle_max_threads.argtypes = []
    return lib


def _p(a: np.ndarray, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


def _prep(weights, bits):
    w = np.ascontiguousarray(weights, dtype=np.int64)
    b = np.ascontiguousarray(bits, dtype=np.uint64)
    return w, b


class COracle:
    """The compiled half of the oracle (``oracle.c``), bound through ctypes.

    The default instance loads ``oracle/_build/liboracle.so``; tests that plant
    mistakes in a copy of ``oracle.c`` load that copy through this class."""

    def __init__(self, path: str | os.PathLike):
        self.path = str(path)
        self.lib = _bind(ctypes.CDLL(self.path))

    def max_threads(self) -> int:
        return int(self.lib.oracle_max_threads())

    def intersection_weights(self, weights, bits) -> np.ndarray:
        """w(I(S)) for every S in [0, 2^m) (int64[2^m]); wI[0] = weight of the union."""
        w, b = _prep(weights, bits)
        m = b.shape[0]
        out = np.zeros(1 << m, dtype=np.int64)
        rc = self.lib.oracle_intersection_weights(m, w.shape[0], _p(w, ctypes.c_int64), _p(b, ctypes.c_uint64),
                                                  _p(out, ctypes.c_int64))
        if rc != 0:
            raise RuntimeError(f"oracle_intersection_weights failed ({rc})")
        return out

    def wI_one(self, weights, bits, S: int) -> int:
        w, b = _prep(weights, bits)
        return int(self.lib.oracle_wI_one(b.shape[0], w.shape[0], _p(w, ctypes.c_int64), _p(b, ctypes.c_uint64),
                                          S))

    def dp(self, wI: np.ndarray, m: int, threads: int = 0):
        """The Sec. 3.1 recurrence: returns (F int64[2^m], split uint32[2^m])."""
        wI = np.ascontiguousarray(wI, dtype=np.int64)
        F = np.zeros(1 << m, dtype=np.int64)
        split = np.zeros(1 << m, dtype=np.uint32)
        rc = self.lib.oracle_dp(m, _p(wI, ctypes.c_int64), _p(F, ctypes.c_int64), _p(split, ctypes.c_uint32),
                                threads)
        if rc != 0:
            raise RuntimeError(f"oracle_dp failed ({rc})")
        return F, split

    def dp_at(self, wI: np.ndarray, F: np.ndarray, m: int, subsets, threads: int = 0):
        """The recurrence's step at the listed subsets, from the tables wI and
        F (int64[2^m]): returns (F int64[count], split uint32[count])."""
        wI = np.ascontiguousarray(wI, dtype=np.int64)
        F = np.ascontiguousarray(F, dtype=np.int64)
        S = np.ascontiguousarray(subsets, dtype=np.uint64)
        if wI.shape[0] != (1 << m) or F.shape[0] != (1 << m) or (S.size and int(S.max()) >= (1 << m)):
            raise ValueError("tables must hold 2^m entries and subsets lie below 2^m")
        Fo = np.zeros(S.shape[0], dtype=np.int64)
        so = np.zeros(S.shape[0], dtype=np.uint32)
        rc = self.lib.oracle_dp_at(m, _p(wI, ctypes.c_int64), _p(F, ctypes.c_int64), _p(S, ctypes.c_uint64),
                                   int(S.shape[0]), _p(Fo, ctypes.c_int64), _p(so, ctypes.c_uint32), threads)
        if rc != 0:
            raise RuntimeError(f"oracle_dp_at failed ({rc})")
        return Fo, so

    def solve(self, weights, bits, threads: int = 0):
        """(OPT, F, wI, split) for a whole instance."""
        m = int(np.asarray(bits).shape[0])
        wI = self.intersection_weights(weights, bits)
        F, split = self.dp(wI, m, threads)
        return int(F[(1 << m) - 1]), F, wI, split

    def recompute(self, weights, bits, F_table: np.ndarray, subsets, threads: int = 0):
        """For each S in ``subsets``: (F(S), split(S), w(I(S))) recomputed from
        ``F_table``'s entries for the proper subsets of S, w(I(S)) from scratch."""
        w, b = _prep(weights, bits)
        m = b.shape[0]
        Ft = np.ascontiguousarray(F_table, dtype=np.int64)
        if Ft.shape[0] != (1 << m):
            raise ValueError("F_table must have 2^m entries")
        Ss = np.ascontiguousarray(subsets, dtype=np.uint64)
        cnt = Ss.shape[0]
        Fo = np.zeros(cnt, dtype=np.int64)
        so = np.zeros(cnt, dtype=np.uint32)
        wo = np.zeros(cnt, dtype=np.int64)
        rc = self.lib.oracle_recompute(m, w.shape[0], _p(w, ctypes.c_int64), _p(b, ctypes.c_uint64),
                                       _p(Ft, ctypes.c_int64), _p(Ss, ctypes.c_uint64), cnt,
                                       _p(Fo, ctypes.c_int64), _p(so, ctypes.c_uint32), _p(wo, ctypes.c_int64),
                                       threads)
        if rc != 0:
            raise RuntimeError(f"oracle_recompute failed ({rc})")
        return Fo, so, wo


def _default() -> COracle:
    global _LIB
    if _LIB is None:
        _LIB = COracle(build())
    return _LIB


def max_threads() -> int:
    return _default().max_threads()


def intersection_weights(weights, bits) -> np.ndarray:
    return _default().intersection_weights(weights, bits)


def wI_one(weights, bits, S: int) -> int:
    return _default().wI_one(weights, bits, S)


def dp(wI: np.ndarray, m: int, threads: int = 0):
    return _default().dp(wI, m, threads)


def solve(weights, bits, threads: int = 0):
    return _default().solve(weights, bits, threads)


def recompute(weights, bits, F_table: np.ndarray, subsets, threads: int = 0):
    return _default().recompute(weights, bits, F_table, subsets, threads)


def dp_at(wI: np.ndarray, F: np.ndarray, m: int, subsets, threads: int = 0):
    return _default().dp_at(wI, F, m, subsets, threads)


# ---------------------------------------------------------------------------
# Pure-Python parts (small inputs)
# ---------------------------------------------------------------------------

def request_sets(weights, bits) -> list[set[int]]:
    n = int(np.asarray(weights).shape[0])
    out = []
    for row in np.asarray(bits, dtype=np.uint64):
        s = set()
        for j, word in enumerate(row.tolist()):
            while word:
                low = word & -word
                x = j * 64 + low.bit_length() - 1
                if x < n:
                    s.add(x)
                word ^= low
        out.append(s)
    return out


def layout(weights, bits, split: np.ndarray):
    """Constructive direction of Thm 1 for the hierarchy encoded by ``split``.

    Node S (|S| >= 2) has children A = split[S] (listed first) and S \\ A.
    At node B the chunks of I(B) \\ I(parent(B)) are emitted in increasing
    chunk id; I(parent(root)) is empty.  Returns (perms, dfs): perms[i] is the
    chunk sequence of request i, dfs the leaves from left to right.
    """
    R = request_sets(weights, bits)
    m = len(R)
    perms: list[list[int]] = [[] for _ in range(m)]
    dfs: list[int] = []

    def members(S):
        return [i for i in range(m) if (S >> i) & 1]

    def inter(S):
        it = members(S)
        acc = set(R[it[0]])
        for i in it[1:]:
            acc &= R[i]
        return acc

    def walk(S, parent_I):
        I = inter(S)
        emit = sorted(I - parent_I)
        for i in members(S):
            perms[i].extend(emit)
        if S & (S - 1) == 0:
            dfs.append(S.bit_length() - 1)
            return
        A = int(split[S])
        if A == 0 or (A & ~S) or A == S:
            raise ValueError(f"split[{S}] = {A} is not a proper subset")
        walk(A, I)
        walk(S ^ A, I)

    walk((1 << m) - 1, set())
    return perms, dfs


def trie_cost(weights, perms) -> int:
    """Eq. (1): the sum of w(chunk(v)) over non-root nodes v of the trie of ``perms``."""
    w = np.asarray(weights)
    root: dict = {}
    cost = 0
    for seq in perms:
        node = root
        for x in seq:
            x = int(x)
            if x not in node:
                node[x] = {}
                cost += int(w[x])
            node = node[x]
    return cost


def brute_force_permutations(weights, bits) -> int:
    """OPT_free by definition: min of eq. (1) over every per-request permutation."""
    R = [sorted(s) for s in request_sets(weights, bits)]
    best = None
    for choice in itertools.product(*[list(itertools.permutations(r)) for r in R]):
        c = trie_cost(weights, choice)
        if best is None or c < best:
            best = c
    return int(best)


def _hierarchies(leaves):
    """Every rooted binary tree with the given leaves, as nested tuples."""
    if len(leaves) == 1:
        yield leaves[0]
        return
    first, rest = leaves[0], leaves[1:]
    # unordered splits: the part holding `first` is one child
    for r in range(0, len(rest)):
        for comb in itertools.combinations(rest, r):
            left = (first,) + comb
            right = tuple(x for x in rest if x not in comb)
            for L in _hierarchies(list(left)):
                for Rt in _hierarchies(list(right)):
                    yield (L, Rt)


def _clusters(tree):
    """(cluster, parent cluster) for every node of a nested-tuple tree."""
    out = []

    def leafset(t):
        if isinstance(t, tuple):
            return leafset(t[0]) | leafset(t[1])
        return frozenset([t])

    def rec(t, parent):
        c = leafset(t)
        out.append((c, parent))
        if isinstance(t, tuple):
            rec(t[0], c)
            rec(t[1], c)

    rec(tree, None)
    return out


def brute_force_hierarchies(weights, bits) -> int:
    """Eq. (2): min over binary hierarchies H of sum_x w(x) t_x(H), where
    t_x(H) counts the maximal clusters of H contained in S_x = {i : x in R_i}."""
    R = request_sets(weights, bits)
    m = len(R)
    w = np.asarray(weights)
    chunks = sorted(set().union(*R)) if R else []
    S_x = {x: frozenset(i for i in range(m) if x in R[i]) for x in chunks}
    best = None
    for tree in _hierarchies(list(range(m))):
        cl = _clusters(tree)
        total = 0
        for x in chunks:
            sx = S_x[x]
            t = sum(1 for c, parent in cl if c <= sx and (parent is None or not parent <= sx))
            total += int(w[x]) * t
        if best is None or total < best:
            best = total
    return int(best)


def brute_force_global_order(weights, bits) -> int:
    """OPT_glob (Sec. 2): every request sorted by one common chunk order."""
    R = request_sets(weights, bits)
    chunks = sorted(set().union(*R)) if R else []
    best = None
    for order in itertools.permutations(chunks):
        rank = {x: r for r, x in enumerate(order)}
        perms = [sorted(r, key=lambda x: rank[x]) for r in R]
        c = trie_cost(weights, perms)
        if best is None or c < best:
            best = c
    return int(best if best is not None else 0)


def global_order_cost(weights, bits, order=None) -> int:
    """Trie cost when every request is sorted by one chunk order (default: chunk id)."""
    R = request_sets(weights, bits)
    if order is None:
        perms = [sorted(r) for r in R]
    else:
        rank = {x: r for r, x in enumerate(order)}
        perms = [sorted(r, key=lambda x: rank[x]) for r in R]
    return trie_cost(weights, perms)


def min_vertex_cover(edges, vertices) -> int:
    """tau(G) by brute force over vertex subsets (Prop 2)."""
    vs = sorted(vertices)
    for size in range(len(vs) + 1):
        for cover in itertools.combinations(vs, size):
            c = set(cover)
            if all(u in c or v in c for u, v in edges):
                return size
    return len(vs)


def spanning_tree_bound(weights, bits) -> int:
    """Sec. 6.3: sum_i w(R_i) - MaxSpanningTree(w(R_i cap R_j)), a lower bound on OPT."""
    R = request_sets(weights, bits)
    w = np.asarray(weights)
    m = len(R)
    wt = lambda s: int(sum(int(w[x]) for x in s))
    total = sum(wt(r) for r in R)
    if m <= 1:
        return total
    # Prim's algorithm for a maximum spanning tree
    in_tree = [False] * m
    best = [-1] * m
    in_tree[0] = True
    for j in range(1, m):
        best[j] = wt(R[0] & R[j])
    mst = 0
    for _ in range(m - 1):
        j = max((j for j in range(m) if not in_tree[j]), key=lambda j: best[j])
        mst += best[j]
        in_tree[j] = True
        for k in range(m):
            if not in_tree[k]:
                best[k] = max(best[k], wt(R[j] & R[k]))
    return total - mst


def radix_cache_cost(weights, perms, order, capacity) -> int:
    """Prefill tokens paid by a radix (prefix) cache with LRU leaf eviction.

    Requests are served in ``order``.  A cached node implies its ancestors are
    cached; to make room, the least recently used leaf that is not an ancestor
    of the node being inserted is evicted (Sec. 8).  Each chunk not found on
    the cached path is computed (its weight is paid) and inserted; if no room
    can be made, the rest of the request is computed without caching."""
    w = np.asarray(weights)
    cached: dict = {}  # prefix tuple -> time of last use
    nchild: dict = {(): 0}  # cached prefix (and the root) -> number of cached children
    used = 0
    clock = 0
    paid = 0
    for i in order:
        seq = tuple(int(x) for x in perms[i])
        for d in range(1, len(seq) + 1):
            key = seq[:d]
            clock += 1
            if key in cached:
                cached[key] = clock
                continue
            need = int(w[key[-1]])
            paid += need
            protected = {seq[:e] for e in range(1, d)}
            while used + need > capacity:
                leaves = [k for k in cached if nchild[k] == 0 and k not in protected]
                if not leaves:
                    break
                victim = min(leaves, key=cached.get)
                del cached[victim]
                del nchild[victim]
                nchild[victim[:-1]] -= 1
                used -= int(w[victim[-1]])
            if used + need > capacity:
                paid += sum(int(w[x]) for x in seq[d:])
                break
            cached[key] = clock
            nchild[key] = 0
            nchild[key[:-1]] += 1
            used += need
    return paid


def loo_free(n: int) -> int:
    """Thm 5: OPT_free(L_n) = n*ceil(log2 n) - 2^ceil(log2 n) + n."""
    c = math.ceil(math.log2(n)) if n > 1 else 0
    return n * c - (1 << c) + n


def loo_glob(n: int) -> int:
    """Thm 5: OPT_glob(L_n) = (n-1)(n+2)/2."""
    return (n - 1) * (n + 2) // 2


def greedy(weights, bits):
    """Agglomerative common-intersection hierarchy (Sec. 6.2; H_g of Thm 6).

    Every request starts as a cluster whose signature is R_i.  Repeatedly the
    two active clusters with the heaviest common signature w(I(A) cap I(B))
    are merged, the merged signature being that intersection.  A cluster is
    held in the slot of its smallest request; ties go to the smallest slot
    pair (a, b), a < b (a reading: the paper leaves ties open).  The merged
    cluster keeps slot a.

    Returns dict(merges=[(a, b, value)], savings, cost = sum_i w(R_i) - savings,
    perms, dfs): the layout walks the hierarchy top-down as in Thm 1 (at each
    node the chunks of I(v) minus I(parent(v)), increasing id), children of a
    merge ordered (slot a, slot b), dfs the leaves from left to right."""
    R = request_sets(weights, bits)
    w = np.asarray(weights)
    m = len(R)
    wt = lambda s: int(sum(int(w[x]) for x in s))
    sig = [set(r) for r in R]
    node = list(range(m))  # current tree node of each slot
    children = {}
    node_sig = {i: frozenset(R[i]) for i in range(m)}
    active = [True] * m
    merges = []
    for t in range(m - 1):
        best = None
        for a in range(m):
            if not active[a]:
                continue
            for b in range(a + 1, m):
                if not active[b]:
                    continue
                v = wt(sig[a] & sig[b])
                if best is None or v > best[2]:
                    best = (a, b, v)
        a, b, v = best
        merges.append(best)
        sig[a] = sig[a] & sig[b]
        active[b] = False
        new = m + t
        children[new] = (node[a], node[b])
        node_sig[new] = frozenset(sig[a])
        node[a] = new
    savings = sum(v for _, _, v in merges)
    total = sum(wt(r) for r in R)
    perms: list[list[int]] = [[] for _ in range(m)]
    dfs: list[int] = []

    def walk(v, parent_sig):
        emit = sorted(node_sig[v] - parent_sig)
        leaves = []
        if v < m:
            perms[v].extend(emit)
            dfs.append(v)
            return [v]
        left, right = children[v]
        for i in _leaves(left, children, m) + _leaves(right, children, m):
            perms[i].extend(emit)
        walk(left, node_sig[v])
        walk(right, node_sig[v])
        return leaves

    if m > 0:
        walk(node[0] if m > 1 else 0, frozenset())
    return dict(merges=merges, savings=savings, cost=total - savings, perms=perms, dfs=dfs)


def _leaves(v, children, m):
    if v < m:
        return [v]
    l, r = children[v]
    return _leaves(l, children, m) + _leaves(r, children, m)


def trie_cost_sorted(weights, perms) -> int:
    """Eq. (1) for many strings: sort them lexicographically; each string adds
    the weight of its suffix after the longest common prefix with its
    predecessor (each trie node is counted once, at the first string that
    reaches it in sorted order)."""
    w = np.asarray(weights)
    seqs = sorted(tuple(int(x) for x in p) for p in perms)
    cost = 0
    prev: tuple = ()
    for sq in seqs:
        l = 0
        while l < len(sq) and l < len(prev) and sq[l] == prev[l]:
            l += 1
        cost += int(sum(int(w[x]) for x in sq[l:]))
        prev = sq
    return cost


def recompute_local(weights, bits, S: int, F_sub) -> tuple[int, int, int]:
    """F(S), split(S) and w(I(S)) for one subset S from a table of S's own
    submasks: F_sub[j] = F(A) where A has the bits of j deposited into the set
    bits of S (j = 0 .. 2^|S| - 1).  Depositing preserves order, so the
    smallest index j is the smallest A; the lowest request of S is bit 0 of j.
    Used to check single entries of tables too large for oracle_dp."""
    F_sub = np.asarray(F_sub, dtype=np.int64)
    k = bin(S).count("1")
    full = (1 << k) - 1
    wi = wI_one(weights, bits, S)
    if k <= 1:
        return (wi if S else 0), 0, wi
    j = np.arange(1, full, 2, dtype=np.int64)  # holds bit 0 (the lowest request), not the whole set
    vals = F_sub[j] + F_sub[full ^ j]
    t = int(np.argmin(vals))  # first minimum = smallest A
    jbest = int(j[t])
    A = 0
    pos = [i for i in range(64) if (S >> i) & 1]
    for q, p in enumerate(pos):
        if (jbest >> q) & 1:
            A |= 1 << p
    return int(vals[t]) - wi, A, wi


def serve_order(perms, arrival=None, window: int = 0) -> list[int]:
    """Thm 7 (Sec. 8): serve requests in the DFS order of the trie of their
    laid-out strings, i.e. sorted lexicographically (a string before its
    extensions).  With ``window`` = W in [1, m), the stream ``arrival`` is cut
    into consecutive windows of W arrivals and each window is sorted on its own
    (the bounded reorder window of Sec. 8.1).  Identical strings keep the
    smaller request index first."""
    m = len(perms)
    arr = list(range(m)) if arrival is None else [int(a) for a in arrival]
    W = m if (window <= 0 or window >= m) else int(window)
    out: list[int] = []
    for lo in range(0, m, max(W, 1)):
        out += sorted(arr[lo:lo + W], key=lambda r: (tuple(int(x) for x in perms[r]), r))
    return out


def radix_cache_costs(weights, perms, order, capacities) -> list[int]:
    """``radix_cache_cost`` for each capacity in ``capacities`` (one simulation each)."""
    return [radix_cache_cost(weights, perms, order, int(c)) for c in capacities]


def pinned_layout(weights, ranked, t: int, C=None):
    """Sec. 7.1: pin the first ``t`` passages of each request's relevance-ranked
    list ``ranked[i]`` at the end of its prompt, in relevance order (rank 1
    first), and lay the remaining passages out freely with the exact
    recurrence (Sec. 3.1) on the reduced request sets.  Returns
    (strings, trie cost by eq. (1))."""
    from paper_2609_13692_gb300 import instances as _inst  # bit packing only

    C = C or _default()
    n = len(weights)
    free = [[int(x) for x in r[t:]] for r in ranked]
    pins = [[int(x) for x in r[:t]] for r in ranked]
    bits = _inst.pack_requests(free, n)
    if len(ranked) == 0:
        return [], 0
    _opt, _F, _wI, split = C.solve(np.asarray(weights, dtype=np.int64), bits)
    perms, _dfs = layout(weights, bits, split)
    seqs = [list(p) + q for p, q in zip(perms, pins)]
    return seqs, trie_cost(weights, seqs)


def brute_force_pinned(weights, ranked, t: int) -> int:
    """Least eq. (1) cost over every permutation of each request's free
    passages, with its top ``t`` fixed at the end in relevance order."""
    free = [sorted(int(x) for x in r[t:]) for r in ranked]
    pins = [[int(x) for x in r[:t]] for r in ranked]
    best = None
    for choice in itertools.product(*[list(itertools.permutations(f)) for f in free]):
        c = trie_cost(weights, [list(p) + q for p, q in zip(choice, pins)])
        best = c if best is None or c < best else best
    return int(best)

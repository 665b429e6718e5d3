"""A model of the pair kernel's window ring (k_dp_pairs in
paper_2609_13692_gb300/csrc/k_dp_blocked.cu), run on random interleavings of
its 8 warps.

Per window pair j of a block's range, every warp: waits for "folded" of pair
j + 1 - 4 and issues its copies of pair j + 1 into that ring slot (they land
later, in any order, each landing one arrival on "full"); waits for "full"
of pair j; runs its shared-row slot of the step, if it has one; runs its
register units on pair j; arrives on "consumed" of pair j; then waits for
"consumed" of pair j - 1, folds that pair's shared-row minima and arrives on
"folded" of pair j - 1.  Pairs 2h and 2h + 1 have 9 slots, numbered
9h .. 9h + 8 and run by warp (number mod 8): four full slots of pair 2h at
step 2h, four of pair 2h + 1 and the merged partial slot of both pairs at
step 2h + 1 (a last pair without a partner runs its own partial slot).  The
merged slot's warp holds back its "consumed" arrival for pair 2h until it
has run that slot.

Checked on every interleaving: no deadlock; every arrival lands in the
barrier phase it is meant for; no parity wait can see two phases pass; every
window read finds its pair in the ring slot; no ring slot is refilled before
all reads of its pair; every shared-row flush of a pair goes to the array
that accumulates that pair and happens before anyone folds it.  The planted
mistakes at the end must each be caught.
"""
import random

import pytest

RING = 4
WARPS = 8


def slots_of_step(j, n):
    """(warp, kind) of the slots run at step j of an n-pair range."""
    h, odd = j >> 1, j & 1
    if odd:
        base, count = 9 * h + 4, 5
    else:
        base, count = 9 * h, (5 if j + 1 == n else 4)
    out = []
    for i in range(count):
        kind = "full" if i < 4 else ("merged" if odd else "lone")
        out.append(((base + i) % WARPS, kind))
    return out


def holds_back(w, j, n):
    """True when warp w arrives on "consumed" of pair j only at step j + 1."""
    return j % 2 == 0 and j + 1 < n and w == (j // 2) % WARPS


def simulate(n, rng, holds_back=holds_back, slots_of_step=slots_of_step):
    bars = {(kind, c): [0, 0] for kind in ("full", "consumed", "folded") for c in range(RING)}
    ring = [None] * RING
    landing = []
    smin_pair = list(range(RING))
    folded_by = {}
    reads, writes = {}, {}
    exp_reads = {p: WARPS for p in range(n)}
    exp_writes = {p: 0 for p in range(n)}
    full, partial = [0] * n, [0] * n
    for j in range(n):
        for _, kind in slots_of_step(j, n):
            for p in ([j - 1, j] if kind == "merged" else [j]):
                assert 0 <= p < n, f"slot of pair {p} outside the range"
                exp_reads[p] += 1
                exp_writes[p] += 1
                if kind == "full":
                    full[p] += 1
                else:
                    partial[p] += 1
    # every pair's 139 shared-row units run once: 4 full slots, 1 partial
    assert full == [4] * n and partial == [1] * n, (full, partial)

    def arrive(key, phase):
        b = bars[key]
        assert b[0] == phase, f"arrival on {key} for phase {phase} while in phase {b[0]}"
        b[1] += 1
        if b[1] == WARPS:
            b[0] += 1
            b[1] = 0

    def passable(key, phase):
        done = bars[key][0]
        assert done <= phase + 1, f"parity wait on {key} for phase {phase} after {done} phases"
        return done > phase

    def fold(w, p):
        assert writes.get(p, 0) == exp_writes[p], f"fold of pair {p} before its slot flushes"
        folded_by.setdefault(p, set()).add(w)
        if len(folded_by[p]) == WARPS:
            smin_pair[p % RING] = p + RING
        arrive(("folded", p % RING), p // RING)

    def program(w):
        def copy(p):
            if p >= RING:
                assert reads.get(p - RING, 0) == exp_reads[p - RING], f"slot refilled with pair {p} too early"
            landing.append(p)

        if n >= 1:
            copy(0)
        yield None
        for j in range(n):
            c = j % RING
            if j + 1 < n:
                if j + 1 >= RING:
                    yield ("wait", ("folded", (j + 1) % RING), (j + 1) // RING - 1)
                copy(j + 1)
                yield None
            yield ("wait", ("full", c), j // RING)
            for ww, kind in slots_of_step(j, n):
                if ww != w:
                    continue
                for p in ([j - 1, j] if kind == "merged" else [j]):
                    assert ring[p % RING] == p, f"slot reads pair {p}, ring holds {ring[p % RING]}"
                    assert smin_pair[p % RING] == p, f"flush of pair {p} into the array of {smin_pair[p % RING]}"
                    reads[p] = reads.get(p, 0) + 1
                    writes[p] = writes.get(p, 0) + 1
                if kind == "merged":
                    arrive(("consumed", (j - 1) % RING), (j - 1) // RING)
            yield None
            assert ring[c] == j, f"units read pair {j}, ring holds {ring[c]}"
            reads[j] = reads.get(j, 0) + 1
            yield None
            if not holds_back(w, j, n):
                arrive(("consumed", c), j // RING)
            yield None
            if j >= 1:
                yield ("wait", ("consumed", (j - 1) % RING), (j - 1) // RING)
                fold(w, j - 1)
                yield None
        if n >= 1:
            yield ("wait", ("consumed", (n - 1) % RING), (n - 1) // RING)
            fold(w, n - 1)
            yield None

    progs = [program(w) for w in range(WARPS)]
    waits = [next(p) for p in progs]
    done = [False] * WARPS
    while True:
        ready = [w for w in range(WARPS) if not done[w] and (waits[w] is None or passable(*waits[w][1:]))]
        choices = ready + (["land"] if landing else [])
        if not choices:
            assert all(done), f"deadlock at n = {n}: {waits}"
            break
        pick = rng.choice(choices)
        if pick == "land":
            p = landing.pop(rng.randrange(len(landing)))
            ring[p % RING] = p
            arrive(("full", p % RING), p // RING)
            continue
        try:
            waits[pick] = next(progs[pick])
        except StopIteration:
            done[pick] = True
    for p in range(n):
        assert reads.get(p, 0) == exp_reads[p] and writes.get(p, 0) == exp_writes[p]


def test_slot_rotation_is_balanced():
    # every step's slots go to distinct warps; over 16 pairs each warp runs 9
    for n in (16, 32):
        count = [0] * WARPS
        for j in range(n):
            ws = [w for w, _ in slots_of_step(j, n)]
            assert len(set(ws)) == len(ws)
            for w in ws:
                count[w] += 1
        assert count == [9 * n // 16] * WARPS
    # 139 units = 4 full slots + 11 lanes per pair; two partial slots fill 22 lanes
    assert 4 * 32 + 11 == 139 and 2 * 11 <= 32


@pytest.mark.parametrize("n", list(range(1, 13)) + [17, 40])
def test_ring_protocol_random_interleavings(n):
    rng = random.Random(1000 + n)
    for _ in range(60):
        simulate(n, rng)


def _caught(**planted):
    rng = random.Random(7)
    try:
        for n in range(1, 12):
            for _ in range(40):
                simulate(n, rng, **planted)
    except AssertionError:
        return True
    return False


def test_planted_protocol_mistakes_are_caught():
    # the merged slot's warp arriving for pair 2h at step 2h, before its flush
    assert _caught(holds_back=lambda w, j, n: False)
    # the arrival held back by a warp other than the merged slot's
    assert _caught(holds_back=lambda w, j, n: j % 2 == 0 and j + 1 < n and w == (j // 2 + 1) % WARPS)

    # the partial slot of a pair without a partner left out
    def no_lone(j, n):
        return [s for s in slots_of_step(j, n) if s[1] != "lone"]

    assert _caught(slots_of_step=no_lone)

    # the merged slot run one step late, at step 2h + 2
    def late(j, n):
        out = [s for s in slots_of_step(j, n) if s[1] != "merged"]
        if j % 2 == 0 and j >= 2:
            out.append(((9 * ((j - 2) >> 1) + 8) % WARPS, "merged"))
        return out

    assert _caught(slots_of_step=late)

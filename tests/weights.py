"""Weight totals of an instance that decide which key width the tiled
kernels use: sum_i w(R_i), and the shared weight, the same sum less the
chunks that exactly one request needs and (for m >= 2) those that every
request needs."""

from __future__ import annotations

import numpy as np


def request_counts(inst) -> np.ndarray:
    """|S_x| for every chunk x: the number of requests that hold it."""
    n = inst.weights.shape[0]
    bits = np.unpackbits(np.ascontiguousarray(inst.bits).view(np.uint8), axis=1, bitorder="little")
    return bits[:, :n].sum(axis=0).astype(np.int64)


def request_weight_sum(inst) -> int:
    return int(sum(int(w) * int(c) for w, c in zip(inst.weights, request_counts(inst))))


def shared_weight(inst) -> int:
    m = inst.m
    return int(sum(int(w) * int(c) for w, c in zip(inst.weights, request_counts(inst)) if 2 <= c < m))


def universal_weight(inst) -> int:
    """u: the weight of the chunks that every one of m >= 2 requests holds."""
    if inst.m < 2:
        return 0
    return int(sum(int(w) for w, c in zip(inst.weights, request_counts(inst)) if c == inst.m))


def private_weights(inst) -> list[int]:
    """pi_i: the weight of the chunks that request i alone holds."""
    cnt = request_counts(inst)
    out = []
    for i in range(inst.m):
        row = np.unpackbits(np.ascontiguousarray(inst.bits[i]).view(np.uint8), bitorder="little")
        out.append(int(sum(int(inst.weights[x]) for x in np.flatnonzero(row[: inst.weights.shape[0]]) if cnt[x] == 1)))
    return out

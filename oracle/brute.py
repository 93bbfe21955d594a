"""Pure-Python brute force of the DGE scores, for tiny inputs only.

TEST INFRASTRUCTURE ONLY.  A second, independent statement of Alg. 1 line B /
App. B in plain Python floats with ``math.fsum`` (exactly rounded sums), used
to pin the C oracle on n <= 64, m <= 4, G <= 2.  It takes the attention
weights of each row as softmax over its visible keys and adds them up, the
most literal form of the definition.
"""
from __future__ import annotations

import math
import struct


def bf16_to_float(bits: int) -> float:
    return struct.unpack("<f", struct.pack("<I", (int(bits) & 0xFFFF) << 16))[0]


def attention_row(q, keys, scale):
    """softmax_j(q . k_j * scale) over the given keys, as a list of floats."""
    logits = [scale * math.fsum(a * b for a, b in zip(q, k)) for k in keys]
    mx = max(logits)
    e = [math.exp(x - mx) for x in logits]
    z = math.fsum(e)
    return [x / z for x in e]


def scores(Q_rows, K_rows, positions, P, scale):
    """raw[j] = sum over rows r with j <= positions[r] of softmax weight of key j.

    Q_rows, K_rows: lists of float vectors; positions: list of ints.
    """
    n = len(K_rows)
    per_pos = [[] for _ in range(P)]
    for q, p in zip(Q_rows, positions):
        last = min(p, n - 1)
        a = attention_row(q, K_rows[:last + 1], scale)
        for j in range(min(last + 1, P)):
            per_pos[j].append(a[j])
    return [math.fsum(v) for v in per_pos]


def max_pool(raw, kernel):
    r = kernel // 2
    P = len(raw)
    return [max(raw[max(0, j - r):min(P, j + r + 1)]) for j in range(P)]


def avg_pool(raw, kernel):
    r = kernel // 2
    P = len(raw)
    return [math.fsum(raw[max(0, j - r):min(P, j + r + 1)]) / kernel for j in range(P)]


def top_positions(values, keep):
    """The ``keep`` positions with the largest values, lower position first on ties, ascending."""
    order = sorted(range(len(values)), key=lambda j: (-values[j], j))
    return sorted(order[:keep])

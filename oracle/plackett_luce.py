"""Exact subset probabilities of weighted sampling without replacement.

TEST INFRASTRUCTURE ONLY (see oracle/roi_oracle.py).

Eq. 1 (Sec. 3.1) gives the probability of an ordered draw y_1..y_K from weights
w as prod_k w_{y_k} / (W - sum_{j<k} w_{y_j}).  Eq. 8 (Sec. 4.2.1) makes the
probability of an unordered N-hot mask the sum of Eq. 1 over every ordering of
its members.  Both are enumerated here by brute force (small M only).
"""
from __future__ import annotations

import itertools

import numpy as np


def ordered_draw_probability(w: np.ndarray, order) -> float:
    """Eq. 1 for one ordered draw."""
    w = np.asarray(w, dtype=np.float64)
    total = float(np.sum(w))
    p = 1.0
    taken = 0.0
    for y in order:
        p *= w[y] / (total - taken)
        taken += w[y]
    return p


def subset_probabilities(w: np.ndarray, N: int) -> dict:
    """Eq. 8: {bitmask of an N-subset: probability}, summing Eq. 1 over orderings."""
    w = np.asarray(w, dtype=np.float64)
    M = w.size
    out = {}
    for subset in itertools.combinations(range(M), N):
        key = sum(1 << i for i in subset)
        out[key] = sum(ordered_draw_probability(w, perm)
                       for perm in itertools.permutations(subset))
    return out

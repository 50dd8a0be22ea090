"""Philox-4x32-10 counter-based generator, written from its published definition.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module; only
``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference legs
of ``bench.py`` may use it.

Reference for the generator: J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw,
"Parallel random numbers: as easy as 1, 2, 3", SC'11, Sec. 4 (the Philox family):
a 4-word counter and a 2-word key; each round multiplies words 0 and 2 by two
fixed odd constants, keeps the 64-bit products as (hi, lo) pairs, and forms the
next counter as (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); the key is bumped by
two Weyl constants after every round.  Ten rounds.

The paper being reproduced (RoI, Algorithm 1) only asks for u ~ Uniform(0, 1);
the counter-based generator is how the noise is made reproducible and never
stored.  Counter layout used throughout this project (both sides implement it
independently):

    key     = (seed & 0xffffffff, seed >> 32)
    counter = (q & 0xffffffff, q >> 32, step, tensor_id),  q = e >> 2
    x_e     = output word (e & 3)

where e is the tensor-global flat element index (row * cols + col, with the
row offset of a row-sliced call added to row).
"""
from __future__ import annotations

import numpy as np

# Round multipliers and key-schedule (Weyl) increments of Philox-4x32 (SC'11).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
PHILOX_ROUNDS = 10

_MASK32 = np.uint64(0xFFFFFFFF)


def _mulhilo(a: int, b: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Full 32x32 -> 64-bit product split into (hi, lo) 32-bit words."""
    p = np.uint64(a) * b.astype(np.uint64)
    return (p >> np.uint64(32)).astype(np.uint32), (p & _MASK32).astype(np.uint32)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Ten Philox-4x32 rounds on arrays of counters; returns the 4 output words.

    All inputs are broadcastable uint32 arrays / scalars.
    """
    c0 = np.asarray(c0, dtype=np.uint32)
    c1 = np.asarray(c1, dtype=np.uint32)
    c2 = np.asarray(c2, dtype=np.uint32)
    c3 = np.asarray(c3, dtype=np.uint32)
    c0, c1, c2, c3 = np.broadcast_arrays(c0, c1, c2, c3)
    k0 = int(k0) & 0xFFFFFFFF
    k1 = int(k1) & 0xFFFFFFFF
    for _ in range(PHILOX_ROUNDS):
        hi0, lo0 = _mulhilo(PHILOX_M0, c0)
        hi1, lo1 = _mulhilo(PHILOX_M1, c2)
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint32(k0), lo1,
                          hi0 ^ c3 ^ np.uint32(k1), lo0)
        k0 = (k0 + PHILOX_W0) & 0xFFFFFFFF
        k1 = (k1 + PHILOX_W1) & 0xFFFFFFFF
    return c0, c1, c2, c3


def noise_words(seed: int, step: int, tensor_id: int, e: np.ndarray) -> np.ndarray:
    """The 32-bit random word x_e for tensor-global element indices ``e``."""
    e = np.asarray(e, dtype=np.uint64)
    q = e >> np.uint64(2)
    w = (e & np.uint64(3)).astype(np.int64)
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    out = philox4x32_10((q & _MASK32).astype(np.uint32),
                        (q >> np.uint64(32)).astype(np.uint32),
                        np.uint32(int(step) & 0xFFFFFFFF),
                        np.uint32(int(tensor_id) & 0xFFFFFFFF),
                        seed & 0xFFFFFFFF, seed >> 32)
    words = np.stack(out, axis=0)            # [4, n]
    return np.take_along_axis(words, w[None, :], axis=0)[0]

"""Pins for the oracle's Philox-4x32-10 and its counter layout.

The pin is an independent implementation: Triton's tl.philox (run through
Triton's CPU interpreter as a library), which follows the same published
definition (Salmon et al., SC'11).
"""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

from oracle.philox import philox4x32_10, noise_words

HERE = os.path.dirname(os.path.abspath(__file__))


def _cases():
    rng = np.random.default_rng(7)
    rows = [[0, 0, 0, 0, 0], [2**64 - 1, 2**32 - 1, 2**32 - 1, 2**32 - 1, 2**32 - 1],
            [1, 1, 0, 0, 0], [0x1234567890ABCDEF, 5, 0, 99, 3]]
    for _ in range(28):
        rows.append([int(rng.integers(0, 2**63)) * 2 + int(rng.integers(0, 2))]
                    + [int(v) for v in rng.integers(0, 2**32, size=4)])
    return rows


def test_philox_matches_triton_library():
    pytest.importorskip("triton")
    rows = _cases()
    env = dict(os.environ, TRITON_INTERPRET="1")
    out = subprocess.run([sys.executable, os.path.join(HERE, "_triton_philox.py"), json.dumps(rows)],
                         capture_output=True, text=True, env=env, timeout=600)
    if out.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + out.stderr[-300:])
    ref = json.loads(out.stdout.strip().splitlines()[-1])
    for (seed, c0, c1, c2, c3), want in zip(rows, ref):
        got = philox4x32_10(c0, c1, c2, c3, seed & 0xFFFFFFFF, seed >> 32)
        assert [int(g) for g in got] == want, (seed, c0, c1, c2, c3)


def test_counter_layout():
    """Element e takes word (e & 3) of the block with counter (e >> 2, step, tensor_id)."""
    seed, step, tid = 0xDEADBEEF12345678, 17, 5
    e = np.array([0, 1, 2, 3, 4, 7, 2**34 + 6], dtype=np.uint64)
    x = noise_words(seed, step, tid, e)
    for ei, xi in zip(e.tolist(), x.tolist()):
        q = ei >> 2
        words = philox4x32_10(q & 0xFFFFFFFF, q >> 32, step, tid, seed & 0xFFFFFFFF, seed >> 32)
        assert int(words[ei & 3]) == xi


def test_streams_differ_by_step_and_tensor():
    e = np.arange(4096, dtype=np.uint64)
    a = noise_words(1, 0, 0, e)
    assert not np.array_equal(a, noise_words(1, 1, 0, e))
    assert not np.array_equal(a, noise_words(1, 0, 1, e))
    assert not np.array_equal(a, noise_words(2, 0, 0, e))
    # 32-bit words look uniform: every bit set about half the time
    bits = ((a[:, None] >> np.arange(32, dtype=np.uint32)) & 1).mean(axis=0)
    assert np.all(np.abs(bits - 0.5) < 0.05)

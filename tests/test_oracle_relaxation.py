"""Pins for the relaxed top-N forward (Sec. 3.2 Eq. 3-4, Sec. 4.2.2 Eq. 11-12, Algorithm 1).

Each check uses something other than the oracle's own formula: a library softmax,
a closed form derived by hand, a log-free weight-space restatement, invariants
and limits.
"""
import numpy as np
import pytest
from scipy.special import softmax

from oracle import roi_oracle as O

NM = [(1, 2), (1, 4), (2, 4), (3, 4), (2, 8), (4, 8), (7, 8), (8, 16), (5, 16), (16, 32), (31, 32)]


def _keys(G, M, scale=1.5, seed=0):
    return np.random.default_rng(seed).normal(0.0, scale, size=(G, M))


@pytest.mark.parametrize("tau", [0.05, 0.3, 1.0, 2.5])
@pytest.mark.parametrize("M", [2, 4, 8, 32])
def test_n1_is_gumbel_softmax(M, tau):
    """N = 1: a single step is softmax(kappa / tau) (Sec. 3.2, Eq. 4)."""
    k = _keys(64, M)
    S = O.relaxed_topn(k, 1, tau)
    assert np.allclose(S, softmax(k / tau, axis=-1), rtol=1e-12, atol=1e-15)


def test_tau1_n2_closed_form():
    """tau = 1, N = 2: alpha^(2) = kappa + log(1 - p) gives
    mu^(2) = p (1 - p) / sum p (1 - p), so S = p + p (1 - p) / (1 - sum p^2), p = softmax(kappa)."""
    for M in (3, 4, 8, 16):
        k = _keys(200, M, seed=M)
        p = softmax(k, axis=-1)
        want = p + p * (1 - p) / (1 - np.sum(p * p, axis=-1, keepdims=True))
        assert np.allclose(O.relaxed_topn(k, 2, 1.0), want, rtol=1e-12, atol=1e-15)


def test_worked_example_s_can_exceed_one():
    """p = (0.6, 0.4, 0, 0), tau = 1, N = 2: S_1 = 0.6 + 0.24 / 0.48 = 1.1 (S_j <= 1 is not an invariant)."""
    with np.errstate(divide="ignore"):
        k = np.log(np.array([[0.6, 0.4, 0.0, 0.0]]))
    S = O.relaxed_topn(k, 2, 1.0)
    assert np.allclose(S, [[1.1, 0.9, 0.0, 0.0]], atol=1e-15)


@pytest.mark.parametrize("tau", [0.1, 0.5, 1.0, 3.0])
@pytest.mark.parametrize("N,M", NM)
def test_weight_space_restatement(N, M, tau):
    """With w = exp(alpha / tau) the update alpha += log(1 - mu) is w <- w * (1 - w / sum w)^(1/tau):
    a log-free second statement of the same recursion (keys kept small so nothing underflows)."""
    k = _keys(50, M, scale=0.3, seed=N * 100 + M)
    w = np.exp(k / tau)
    S = np.zeros_like(w)
    for _ in range(N):
        mu = w / w.sum(axis=-1, keepdims=True)
        S += mu
        w = w * (1.0 - mu) ** (1.0 / tau)
    assert np.allclose(O.relaxed_topn(k, N, tau), S, rtol=1e-10, atol=1e-13)


@pytest.mark.parametrize("N,M", NM)
def test_sum_is_n_and_bounds(N, M):
    """Each mu^(k) is a softmax, so sum_j S_j = N; 0 <= S_j <= N."""
    for tau in (0.05, 0.7, 1.0, 4.0):
        k = _keys(300, M, scale=3.0, seed=M + N)
        S = O.relaxed_topn(k, N, tau)
        assert np.allclose(S.sum(axis=-1), N, rtol=0, atol=1e-12 * N)
        assert np.all(S >= 0) and np.all(S <= N + 1e-12)


@pytest.mark.parametrize("N,M", [(1, 4), (2, 4), (3, 4), (4, 8), (8, 16), (16, 32)])
def test_tau_to_zero_is_hard_topn(N, M):
    """tau -> 0: every softmax becomes one-hot and S becomes the hard top-N of the keys."""
    rng = np.random.default_rng(N + M)
    # distinct keys, adjacent gaps >= 0.05
    k = np.stack([rng.permutation(M) * 0.05 + rng.normal(0, 1) for _ in range(100)])
    S = O.relaxed_topn(k, N, 1e-3)
    assert np.allclose(S, O.hard_topn(k, N).astype(float), atol=1e-12)


def test_shift_invariance_and_permutation_equivariance():
    k = _keys(100, 8, seed=3)
    S = O.relaxed_topn(k, 3, 0.4)
    assert np.allclose(O.relaxed_topn(k + 7.25, 3, 0.4), S, rtol=1e-12, atol=1e-14)
    perm = np.random.default_rng(1).permutation(8)
    assert np.allclose(O.relaxed_topn(k[:, perm], 3, 0.4), S[:, perm], rtol=1e-12, atol=1e-14)


def test_wide_key_gaps_stay_exact():
    """Gaps far beyond float range of exp(): log(1 - mu) is taken in log space, so the
    top key re-enters at tau = 1 with the weight of all others (no epsilon clamp)."""
    k = np.array([[400.0, 0.0, -10.0, -20.0]])
    S = O.relaxed_topn(k, 2, 1.0)
    # step 1 picks item 0; alpha_0 becomes LSE(0, -10, -20) ~ 0, so step 2 splits ~evenly
    a0 = np.logaddexp.reduce([0.0, -10.0, -20.0])
    p2 = softmax(np.array([a0, 0.0, -10.0, -20.0]))
    assert np.allclose(S, [[1.0 + p2[0], p2[1], p2[2], p2[3]]], atol=1e-12)
    assert np.allclose(O.relaxed_topn(k, 2, 0.1), [[1.0, 1.0, 0.0, 0.0]], atol=1e-12)


def test_fp32_run_tracks_fp64():
    k = _keys(2000, 8, scale=1.0, seed=11)
    for N, tau in ((4, 0.5), (2, 1.0), (7, 0.2)):
        s64 = O.relaxed_topn(k, N, tau)
        s32 = O.relaxed_topn(k.astype(np.float32), N, tau, dtype=np.float32)
        assert s32.dtype == np.float32
        assert np.max(np.abs(s32 - s64)) < 2e-5

"""Plants plausible mistakes in the oracle (on the CPU, via monkeypatch) and checks
that independent pins catch each one: a dropped exclusion, a misplaced tau, a
wrong sign in the backward, a wrong sign in the Gumbel transform."""
import numpy as np
import pytest
from scipy import stats
from scipy.special import softmax

from oracle import roi_oracle as O


def _closed_form_ok():
    k = np.random.default_rng(0).normal(0, 1.5, size=(50, 4))
    p = softmax(k, axis=-1)
    want = p + p * (1 - p) / (1 - np.sum(p * p, axis=-1, keepdims=True))
    return np.allclose(O.relaxed_topn(k, 2, 1.0), want, rtol=1e-10)


def _weight_space_ok(tau=0.5):
    k = np.random.default_rng(1).normal(0, 0.3, size=(20, 8))
    w, S = np.exp(k / tau), np.zeros((20, 8))
    for _ in range(3):
        mu = w / w.sum(axis=-1, keepdims=True)
        S += mu
        w = w * (1 - mu) ** (1 / tau)
    return np.allclose(O.relaxed_topn(k, 3, tau), S, rtol=1e-10)


def _fd_ok():
    rng = np.random.default_rng(2)
    k, c = rng.normal(size=(10, 4)), rng.normal(size=(10, 4))
    _, hist = O.relaxed_topn(k, 2, 0.7, return_history=True)
    g = O.relaxed_topn_backward(hist, c, 0.7)
    fd = np.zeros_like(k)
    for j in range(4):
        kp, km = k.copy(), k.copy()
        kp[:, j] += 1e-6
        km[:, j] -= 1e-6
        fd[:, j] = (np.sum(c * O.relaxed_topn(kp, 2, 0.7), -1) - np.sum(c * O.relaxed_topn(km, 2, 0.7), -1)) / 2e-6
    return np.allclose(g, fd, rtol=1e-5, atol=1e-8)


def test_pins_pass_on_correct_oracle():
    assert _closed_form_ok() and _weight_space_ok() and _fd_ok()


def test_dropped_exclusion_is_caught(monkeypatch):
    monkeypatch.setattr(O, "_lse_excluding_each", lambda ar, z: np.repeat(O._lse(ar, z)[:, None], z.shape[1], 1))
    assert not _closed_form_ok()


def test_misplaced_tau_is_caught(monkeypatch):
    real = O._lse_excluding_each
    # alpha += log(1 - mu) / tau instead of alpha += log(1 - mu): scale the correction
    monkeypatch.setattr(O, "_lse_excluding_each",
                        lambda ar, z: (real(ar, z) - O._lse(ar, z)[:, None]) * 2.0 + O._lse(ar, z)[:, None])
    assert not _weight_space_ok(0.5)


def test_backward_sign_is_caught(monkeypatch):
    real_einsum = np.einsum

    def flipped(spec, *ops, **kw):
        out = real_einsum(spec, *ops, **kw)
        return -out if spec == "gi,gil->gl" else out

    monkeypatch.setattr(O.np, "einsum", flipped)
    assert not _fd_ok()


def test_gumbel_sign_is_caught(monkeypatch):
    real = O.gumbel_from_uniform
    monkeypatch.setattr(O, "gumbel_from_uniform", lambda u, dtype=np.float64: -real(u, dtype))
    g = O.gumbel_noise(3, 0, 0, 300, 300)
    assert stats.kstest(g, lambda x: np.exp(-np.exp(-x))).pvalue < 1e-6

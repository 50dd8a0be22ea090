"""Pins for the hand-derived backward of the relaxation (logit gradients).

Checked against central finite differences of the float64 forward (noise held
fixed) and against torch.autograd (float64) through a plain restatement of the
forward.
"""
import numpy as np
import pytest

from oracle import roi_oracle as O
from workloads import bf16_bits, make_inputs


def _fd_grad(kappa, c, N, tau):
    """Central differences of L(kappa) = sum c * S(kappa)."""
    G, M = kappa.shape
    grad = np.zeros_like(kappa)
    for j in range(M):
        h = 1e-6 * np.maximum(1.0, np.abs(kappa[:, j]))
        kp, km = kappa.copy(), kappa.copy()
        kp[:, j] += h
        km[:, j] -= h
        lp = np.sum(c * O.relaxed_topn(kp, N, tau), axis=-1)
        lm = np.sum(c * O.relaxed_topn(km, N, tau), axis=-1)
        grad[:, j] = (lp - lm) / (2 * h)
    return grad


@pytest.mark.parametrize("N,M,tau", [(1, 4, 1.0), (2, 4, 1.0), (2, 4, 0.1), (3, 4, 0.7), (4, 8, 0.5),
                                     (2, 8, 1.0), (8, 16, 0.2), (16, 32, 0.2), (5, 8, 2.0)])
def test_backward_matches_central_differences(N, M, tau):
    rng = np.random.default_rng(N * 37 + M)
    kappa = rng.normal(0, 1.0, size=(40, M))
    c = rng.normal(0, 1.0, size=(40, M))
    _, hist = O.relaxed_topn(kappa, N, tau, return_history=True)
    g = O.relaxed_topn_backward(hist, c, tau)
    fd = _fd_grad(kappa, c, N, tau)
    scale = np.max(np.abs(fd), axis=-1, keepdims=True) + 1e-300
    assert np.max(np.abs(g - fd) / scale) < 1e-6


@pytest.mark.parametrize("N,M,tau", [(2, 4, 1.0), (4, 8, 0.5), (8, 16, 0.2), (3, 8, 0.3)])
def test_backward_matches_torch_autograd(N, M, tau):
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    kappa = rng.normal(0, 1.0, size=(64, M))
    c = rng.normal(0, 1.0, size=(64, M))
    kt = torch.tensor(kappa, dtype=torch.float64, requires_grad=True)
    alpha, S = kt, torch.zeros_like(kt)
    for _ in range(N):
        mu = torch.softmax(alpha / tau, dim=-1)
        S = S + mu
        alpha = alpha + torch.log(1 - mu)
    (S * torch.tensor(c)).sum().backward()
    _, hist = O.relaxed_topn(kappa, N, tau, return_history=True)
    g = O.relaxed_topn_backward(hist, c, tau)
    assert np.allclose(g, kt.grad.numpy(), rtol=1e-9, atol=1e-12)


def test_backward_wide_gaps_finite_and_consistent():
    kappa = np.array([[200.0, 0.0, -1.0, -3.0], [0.0, -150.0, -151.0, 40.0]])
    c = np.array([[0.3, -1.0, 2.0, 0.5], [1.0, 2.0, -0.5, 0.1]])
    for tau in (1.0, 0.3):
        _, hist = O.relaxed_topn(kappa, 2, tau, return_history=True)
        g = O.relaxed_topn_backward(hist, c, tau)
        assert np.all(np.isfinite(g))
        fd = _fd_grad(kappa, c, 2, tau)
        assert np.allclose(g, fd, rtol=1e-5, atol=1e-7)
    # gradients of a soft N-hot vector sum to zero per group (shift invariance)
    assert np.allclose(g.sum(axis=-1), 0.0, atol=1e-9)


@pytest.mark.parametrize("lam", [1.0, 0.5])
def test_mask_bwd_end_to_end_fd(lam):
    """Whole op: dL/dphi for L = sum dWm * W * S(phi), noise regenerated from (seed, step)."""
    W, phi, dWm = make_inputs(8, 32, "logw", seed=9)
    phi = phi.numpy()
    Wb, dWb = bf16_bits(W), bf16_bits(dWm)
    N, M, tau = 2, 4, 0.8
    out = O.mask_bwd(phi, Wb, dWb, N, M, tau, seed=11, step=3, tensor_id=2, lam=lam)
    c = (O.bf16_to_f32(dWb).astype(np.float64) * O.bf16_to_f32(Wb)).ravel()
    g = O.gumbel_noise(11, 3, 2, 8, 32)

    def loss(p):
        k = O.perturbed_keys(p.ravel(), g, lam).reshape(-1, M)
        return np.sum(c.reshape(-1, M) * O.relaxed_topn(k, N, tau))

    p0 = phi.astype(np.float64)
    fd = np.zeros(p0.size)
    for i in range(p0.size):
        h = 1e-5
        pp, pm = p0.ravel().copy(), p0.ravel().copy()
        pp[i] += h
        pm[i] -= h
        fd[i] = (loss(pp) - loss(pm)) / (2 * h)
    got = out["dlogits"].ravel()
    assert np.max(np.abs(got - fd)) < 1e-6 * np.max(np.abs(fd))
    # dW = bf16(dWm * S)
    assert np.array_equal(out["dW"].ravel(), O.bf16_product(dWb.ravel(), out["soft"].ravel()))

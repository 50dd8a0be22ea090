"""Pins for the logits optimizer step and the temperature schedule of the oracle.

* AdamW (the optimizer of Sec. 5.1, beta = (0.9, 0.95), weight decay 0.05): three
  steps against torch.optim.AdamW in float64, a library implementation.
* Eq. 13 annealing: endpoints, the clamp at the final value, the geometric midpoint.
"""
import numpy as np
import pytest

from oracle import roi_oracle as O


def test_adamw_matches_torch_optim():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    phi0 = rng.normal(0, 0.01, size=257)
    grads = [rng.normal(0, 1e-5, size=257) for _ in range(3)]
    p = torch.tensor(phi0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([p], lr=1e-3, betas=(0.9, 0.95), eps=1e-8, weight_decay=0.05)
    phi, m, v = phi0.copy(), np.zeros(257), np.zeros(257)
    for t, g in enumerate(grads, start=1):
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        phi, m, v = O.adamw_step(phi, g, m, v, 1e-3, 0.9, 0.95, 1e-8, 0.05, t)
        assert np.allclose(phi, p.detach().numpy(), rtol=1e-13, atol=1e-18)
    state = opt.state[p]
    assert np.allclose(m, state["exp_avg"].numpy(), rtol=1e-13)
    assert np.allclose(v, state["exp_avg_sq"].numpy(), rtol=1e-13)


def test_adamw_float32_mode_rounds_like_float64_to_single_precision():
    rng = np.random.default_rng(4)
    phi, g = rng.normal(0, 0.01, 64), rng.normal(0, 1e-5, 64)
    m, v = rng.normal(0, 1e-6, 64), rng.uniform(0, 1e-10, 64)
    a = O.adamw_step(phi, g, m, v, 1e-3, 0.9, 0.95, 1e-8, 0.05, 7)
    b = O.adamw_step(phi, g, m, v, 1e-3, 0.9, 0.95, 1e-8, 0.05, 7, dtype=np.float32)
    for x, y in zip(a, b):
        assert y.dtype == np.float32
        assert np.allclose(x, y, rtol=1e-5, atol=1e-12)


def test_anneal_schedule_eq13():
    tau = O.anneal(1.0, 0.05, [0, 750, 1500, 2000], 1500)
    assert tau[0] == 1.0
    assert np.isclose(tau[1], np.sqrt(0.05), rtol=1e-14)    # geometric midpoint
    assert np.isclose(tau[2], 0.05, rtol=1e-14) and tau[3] == 0.05
    lam = O.anneal(1.0, 0.002, np.arange(0, 2001), 1500)
    assert np.all(np.diff(lam) <= 0) and lam[-1] == 0.002 and lam[0] == 1.0

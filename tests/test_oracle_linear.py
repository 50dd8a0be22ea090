"""Pins for the oracle's masked linear forward (Eq. 5: the layer's product with
W (.) S), independent of its own formula:

* a hand-worked case in the tau -> 0 limit (tests/golden/masked_linear_hand.json);
* identity tokens read back Wm transposed (catches a transposed operand or index);
* tau -> 0 with random inputs equals the brute-force product with the hard
  Gumbel-top-N mask, summed term by term in plain Python;
* torch.nn.functional.linear in float64 on the same decoded values;
* one call over T tokens equals T single-token calls (rows of Y independent).
"""
import json
import os

import numpy as np
import pytest

from oracle import roi_oracle as O
from workloads import bf16_bits, make_inputs, make_tokens

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "masked_linear_hand.json")


def _bits(a):
    import torch
    return bf16_bits(torch.tensor(a, dtype=torch.float32).to(torch.bfloat16))


def test_hand_worked_case():
    g = json.load(open(GOLDEN))
    out = O.masked_linear_fwd(_bits(g["X"]), np.array(g["logits"], np.float32), _bits(g["W"]), g["N"], g["M"],
                              g["tau"], g["seed"], g["step"])
    assert np.array_equal(O.bf16_to_f32(out["Wm"]), np.array(g["Wm"], np.float32))
    assert np.array_equal(out["Y"], np.array(g["Y"]))


def test_identity_tokens_read_back_wm_transposed():
    W, phi, _ = make_inputs(6, 16, "normal", 4)
    X = np.eye(16, dtype=np.float32)
    out = O.masked_linear_fwd(_bits(X), phi.numpy(), bf16_bits(W), 2, 4, 0.8, 9, 2)
    assert np.array_equal(out["Y"], O.bf16_to_f32(out["Wm"]).astype(np.float64).T)


def test_tau_to_zero_is_the_hard_masked_product():
    W, phi, _ = make_inputs(5, 24, "normal", 6)
    X = make_tokens(3, 24, 6)
    Wb, Xb = bf16_bits(W), bf16_bits(X)
    N, M, seed, step = 4, 8, 2, 5
    out = O.masked_linear_fwd(Xb, phi.numpy(), Wb, N, M, 1e-4, seed, step)
    hard = O.mask_fwd(phi.numpy(), Wb, N, M, 1.0, seed, step)["hard"]
    gap = O.topn_key_gap(O.mask_fwd(phi.numpy(), Wb, N, M, 1.0, seed, step)["keys"].reshape(-1, M), N)
    assert gap.min() > 1e-2  # the limit is exact only away from ties
    w = O.bf16_to_f32(Wb).astype(np.float64)
    x = O.bf16_to_f32(Xb).astype(np.float64)
    for t in range(3):
        for r in range(5):
            want = 0.0
            for c in range(24):
                if hard[r, c]:
                    want += x[t, c] * w[r, c]
            assert out["Y"][t, r] == pytest.approx(want, rel=1e-12, abs=1e-15)


def test_matches_torch_linear_float64():
    torch = pytest.importorskip("torch")
    W, phi, _ = make_inputs(12, 64, "logw", 8)
    X = make_tokens(7, 64, 8)
    out = O.masked_linear_fwd(bf16_bits(X), phi.numpy(), bf16_bits(W), 2, 4, 1.0, 1, 1)
    Wm = torch.tensor(O.bf16_to_f32(out["Wm"]), dtype=torch.float64)
    want = torch.nn.functional.linear(X.to(torch.float64), Wm).numpy()
    np.testing.assert_allclose(out["Y"], want, rtol=1e-13, atol=1e-18)


def test_tokens_are_independent():
    W, phi, _ = make_inputs(4, 32, "normal", 10)
    X = make_tokens(5, 32, 10)
    Wb, Xb = bf16_bits(W), bf16_bits(X)
    full = O.masked_linear_fwd(Xb, phi.numpy(), Wb, 2, 4, 0.5, 4, 4, lam=0.7)["Y"]
    for t in range(5):
        one = O.masked_linear_fwd(Xb[t:t + 1], phi.numpy(), Wb, 2, 4, 0.5, 4, 4, lam=0.7)["Y"]
        assert np.array_equal(one[0], full[t])

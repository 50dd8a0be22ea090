"""Pins for hard top-N, the deployment export, bit packing and bf16 rounding."""
import numpy as np
import pytest

from oracle import plackett_luce as PL
from oracle import roi_oracle as O


def test_export_is_most_probable_subset():
    """argtop_N(phi) is the mode of the mask law of Eq. 8 (brute force over subsets)."""
    rng = np.random.default_rng(0)
    for M, N in ((4, 1), (4, 2), (4, 3), (8, 2), (8, 4), (6, 3)):
        for _ in range(20):
            phi = rng.normal(0, 1.0, size=M)
            probs = PL.subset_probabilities(np.exp(phi), N)
            mode = max(probs, key=probs.get)
            hard = O.hard_mask_export(phi[None, :].astype(np.float32), N, M)["hard"][0]
            assert sum(1 << i for i in range(M) if hard[i]) == mode


def test_tie_and_nan_rules():
    k = np.array([[1.0, 1.0, 1.0, 0.0],        # ties: lower index wins
                  [np.nan, 0.0, -1.0, 5.0],    # NaN ranks as -inf
                  [-np.inf, -np.inf, -np.inf, -np.inf],
                  [-0.0, 0.0, -0.0, 0.0]])     # -0 == +0: index order
    h = O.hard_topn(k, 2)
    assert h.tolist() == [[True, True, False, False], [False, True, False, True],
                          [True, True, False, False], [True, True, False, False]]


def test_export_pruned_weights():
    phi = np.array([[0.1, 0.9, -2.0, 0.5, 3.0, 2.0, 1.0, 0.0]], dtype=np.float32)
    W = np.array([[0x3F80, 0xBF80, 0x4000, 0x8000, 0x1234, 0xFFFF, 0x7F80, 0x0001]], dtype=np.uint16)
    out = O.hard_mask_export(phi, 2, 4, W)
    assert out["hard"].tolist() == [[False, True, False, True, True, True, False, False]]
    assert out["W_pruned"].tolist() == [[0, 0xBF80, 0, 0x8000, 0x1234, 0xFFFF, 0, 0]]


def test_bit_packing_order():
    m = np.zeros(70, dtype=bool)
    m[[0, 33, 69]] = True
    w = O.pack_bits(m)
    assert w.tolist() == [1, 2, 1 << 5]
    assert np.array_equal(O.unpack_bits(w, 70), m)


def test_bf16_rne_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    x = np.concatenate([rng.normal(0, 1, 20000), rng.normal(0, 1e-38, 2000), rng.normal(0, 1e38, 2000),
                        [0.0, -0.0, np.inf, -np.inf, 3.3895e38, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8]])
    x = x.astype(np.float32)
    # exact ties: bit patterns with the low half = 0x8000
    ties = (rng.integers(0, 2 ** 16, 500).astype(np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, ties[np.isfinite(ties)]])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.f32_to_bf16_rne(x), want)
    assert np.isnan(O.bf16_to_f32(O.f32_to_bf16_rne(np.array([np.nan], np.float32)))).all()
    back = O.bf16_to_f32(want)
    assert np.array_equal(back, torch.from_numpy(want.view(np.int16)).view(torch.bfloat16).float().numpy())

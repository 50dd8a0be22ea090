"""Pins for the uniform map and the Gumbel noise (Algorithm 1; Sec. 3.2, Eq. 2)."""
from fractions import Fraction

import numpy as np
from scipy import stats

from oracle import roi_oracle as O


def test_uniform_map_exact_and_open_interval():
    x = np.array([0, 1 << 9, 0xFFFFFFFF, 0x80000000, 511], dtype=np.uint32)
    u = O.uniform_from_word(x)
    for xi, ui in zip(x.tolist(), u.tolist()):
        assert Fraction(ui) == (Fraction(xi >> 9) + Fraction(1, 2)) * Fraction(1, 2**23)
        assert 0.0 < ui < 1.0
        assert float(np.float32(ui)) == ui      # exactly representable in float32
    assert u[0] == 2.0 ** -24 and u[2] == 1.0 - 2.0 ** -24


def test_gumbel_distribution_ks():
    """g = -log(-log u) from the Philox stream is Gumbel(0,1): CDF exp(-exp(-x))."""
    g = O.gumbel_noise(seed=3, step=0, tensor_id=0, rows=1000, cols=1000)
    res = stats.kstest(g, lambda x: np.exp(-np.exp(-x)))
    assert res.pvalue > 1e-3
    assert abs(np.mean(g) - np.euler_gamma) < 5e-3          # mean of Gumbel(0,1)
    assert abs(np.var(g) - np.pi ** 2 / 6) < 1e-2           # variance pi^2/6


def test_gumbel_endpoints():
    u = O.uniform_from_word(np.array([0, 0xFFFFFFFF], dtype=np.uint32))
    g = O.gumbel_from_uniform(u)
    assert np.isclose(g[0], -np.log(24 * np.log(2.0)))
    assert np.isclose(g[1], -np.log(-np.log1p(-2.0 ** -24)), rtol=1e-12)


def test_gumbel_fp32_is_rounded_fp64():
    g64 = O.gumbel_noise(5, 2, 1, 64, 64)
    g32 = O.gumbel_noise(5, 2, 1, 64, 64, dtype=np.float32)
    assert g32.dtype == np.float32
    # two correctly rounded logs: |error| <= half an ulp of g plus the relative
    # rounding of E = -log u carried through the outer log (2^-24 absolute)
    bound = 0.5 * np.spacing(np.abs(g64).astype(np.float32)) + 2.0 ** -24 * 1.01
    assert np.all(np.abs(g32.astype(np.float64) - g64) <= bound)


def test_keys_with_lambda():
    """Sec. 4.2.3: sampling temperature lambda scales the logits, kappa = phi/lambda + g."""
    phi = np.array([0.5, -1.0, 2.0, 0.0], dtype=np.float32)
    g = np.array([0.1, 0.2, -0.3, 1.0])
    k = O.perturbed_keys(phi, g, lam=0.25)
    assert np.allclose(k, phi.astype(np.float64) * 4.0 + g)

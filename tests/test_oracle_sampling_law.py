"""The hard mask from Gumbel-top-N of phi + g draws N of M without replacement with
the weighted-reservoir law: Eq. 1 summed over orderings (Eq. 8), Theorem 1.

Frequencies over 10^6 seeded groups are compared with the brute-force enumeration
by a chi-square test; the enumeration itself is pinned by closed cases.
"""
import math

import numpy as np
import pytest
from scipy import stats

from oracle import plackett_luce as PL
from oracle import roi_oracle as O


def test_enumerator_closed_cases():
    w = np.array([1.0, 2.0, 3.0, 4.0])
    p1 = PL.subset_probabilities(w, 1)
    assert np.allclose([p1[1 << i] for i in range(4)], w / w.sum())
    for N in (1, 2, 3):
        assert math.isclose(sum(PL.subset_probabilities(w, N).values()), 1.0, rel_tol=1e-12)
    p = PL.subset_probabilities(np.ones(8), 3)
    assert np.allclose(list(p.values()), 1.0 / math.comb(8, 3))
    # N = M - 1: leaving out item j has probability ... complement of the single draw law
    p3 = PL.subset_probabilities(w, 3)
    # ordered draw of two items (a then b): w_a/W * w_b/(W - w_a)
    assert math.isclose(PL.ordered_draw_probability(w, (3, 0)), 4 / 10 * 1 / 6)
    assert len(p3) == 4


@pytest.mark.parametrize("N,M,G", [(2, 4, 1_000_000), (4, 8, 1_000_000), (2, 8, 400_000)])
def test_gumbel_topn_subset_frequencies(N, M, G):
    rng = np.random.default_rng(N * 10 + M)
    phi = rng.normal(0.0, 0.6, size=M)
    g = O.gumbel_noise(seed=1234 + M, step=N, tensor_id=0, rows=G, cols=M)
    keys = O.perturbed_keys(np.tile(phi, G), g).reshape(G, M)
    hard = O.hard_topn(keys, N)
    assert np.all(hard.sum(axis=1) == N)
    codes = (hard.astype(np.int64) << np.arange(M)).sum(axis=1)
    probs = PL.subset_probabilities(np.exp(phi), N)
    subsets = sorted(probs)
    counts = np.array([np.count_nonzero(codes == s) for s in subsets])
    expected = np.array([probs[s] for s in subsets]) * G
    assert counts.sum() == G
    chi2 = np.sum((counts - expected) ** 2 / expected)
    pval = stats.chi2.sf(chi2, df=len(subsets) - 1)
    assert pval > 1e-3, (chi2, pval)

"""CPU oracle for the RoI mask-learning hot path.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py, never by the product package.
"""
from .philox import philox4x32_10, noise_words  # noqa: F401
from . import roi_oracle, plackett_luce  # noqa: F401

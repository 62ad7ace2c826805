"""Host-side helpers of bench.py (no GPU): the mean accepted tokens reported from an
acceptance histogram."""

import numpy as np

import bench
from oracle import alr_oracle as orc


def test_mat_from_histogram_matches_per_anchor_mean():
    """MAT (Sec. 4) is the mean over anchors of accepted slots + 1; from the histogram of the
    oracle's accepted lengths it must equal the direct per-anchor mean."""
    rng = np.random.default_rng(4)
    A, B = 300, 16
    am_t = rng.integers(0, 3, A * B)
    am_d = np.where(rng.random(A * B) < 0.8, am_t, rng.integers(0, 3, A * B))
    acc, hist = orc.accept_len(am_d, am_t, B)
    assert abs(bench.mean_accepted_tokens(hist.tolist()) - (acc.mean() + 1.0)) < 1e-12
    assert bench.mean_accepted_tokens([0] * (B + 1)) is None
    assert bench.mean_accepted_tokens([5, 0, 0]) == 1.0

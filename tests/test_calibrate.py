"""The library's calibration fits (nr_calib_fit_s_max, nr_calib_fit_gate:
host code, run here without a GPU) against the oracle's loops on random
inputs: ties in x and in y, missing targets, every bin count."""
import numpy as np
import pytest

from oracle import calibrate as oc
from paper_2608_15438_gb300 import calibrate as pc


def test_fits_match_oracle():
    rng = np.random.default_rng(11)
    for trial in range(60):
        n = int(rng.integers(1, 400))
        x = rng.gamma(2.0, 1.0, n).astype(np.float32)
        if trial % 3 == 0:
            x = np.round(x * 2) / 2                     # ties in x
        y = (rng.gamma(1.2, 1.0, n) * (1 + x)).astype(np.float32)
        if trial % 4 == 0:
            y = np.round(y)                             # ties in y
        miss = rng.random(n) < 0.15
        x[miss], y[miss] = np.nan, np.nan
        for bins in (1, 3, 16):
            for q in (0.0, 0.5, 0.9, 0.95, 0.99, 1.0):
                want = oc.fit_gate(x, y, bins, q)
                got = pc.fit_gate(x, y, bins, q)
                if want is None:
                    assert got is None
                    continue
                assert np.array_equal(np.array(got[0], np.float32), np.array(want[0], np.float32))
                assert np.array_equal(np.array(got[1], np.float32), np.array(want[1], np.float32))
        scores = rng.gamma(1.0, 0.1, (max(1, n // 10), 10)).astype(np.float32)
        scores[rng.random(scores.shape) < 0.2] = np.nan
        for cov in (0.0, 0.5, 0.9, 0.99, 1.0):
            assert pc.fit_s_max(scores, cov) == oc.fit_s_max(scores, cov)


def test_fit_arguments():
    with pytest.raises(ValueError):
        pc.fit_gate(np.ones(3, np.float32), np.ones(3, np.float32), 17, 0.9)
    assert pc.fit_s_max(np.full((2, 3), np.nan, np.float32), 0.9) == (None, 0.0, 0.0)

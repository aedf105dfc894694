"""The oracle's calibration of S_max and M(x) (Sec. 3.4), pinned: the target
bucket score equals the bucket enumeration's own key cost for every probed
code (whose order is pinned by the hand-enumerated b = 4 list and the
all-subsets sort); locations, x, y and scores on the hand-worked index whose
fp32 distances are exact; the fits on hand-computed quantile bins."""
import math

import numpy as np
import pytest

import oracle
from oracle import calibrate as oc
from test_oracle_select_seq import hand_index


def test_bucket_score_is_the_enumeration_cost(tmp_path):
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, 20_000)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    path = str(tmp_path / "t.nrix")
    build_index(config(w.dtype, w.dim, w.hidden, 10, 8, 8), base, (W1, b1, W2[:10], b2[:10]), path)
    ix = oracle.Index(path)
    lg = ix.encode(synth.queries(w, 20))
    tau = ix.tau()
    for i in range(len(lg)):
        codes, keys, _ = oracle.probe_list(lg[i], tau, 1024, oracle.params())
        cost = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
        assert len(codes) == 1024
        for c, s in zip(codes, cost):
            assert oc.bucket_score(lg[i], tau, int(c)) == s


def test_hand_worked_locations_and_observations(tmp_path):
    """Hand index (logit (0, 0), u0 = 0, scores 0, 0.5, 0.5, 1 for codes 0..3;
    row r in cluster r). Query 0 targets rows 1 (bucket 0: clusters 0, 1),
    2 (bucket 1: the singleton cluster 2) and 4 (bucket 2: clusters 3..5):
    x = min(1, 4, 0.25, 9, 0.25) = 0.25, the farthest gated target is row 4
    (d 9): y = 8.75. Query 1 targets rows 9 and 6 (bucket 3: clusters 6..9):
    x = 0.0625, y = 16 - 0.0625. Query 2 targets only the singleton: no x."""
    ix = hand_index(tmp_path)
    assert oc.locate(ix, [1, 2, 4, 9, 6, 42, -1]) == [
        (1, 0, 0, 2), (2, 1, 2, 1), (4, 2, 3, 3), (9, 3, 6, 4), (6, 3, 6, 4), (-1, -1, -1, 0),
        (-1, -1, -1, 0)]
    logits = np.zeros((3, 2), np.float32)
    targets = np.array([[1, 2, 4], [9, 6, -1], [2, -1, -1]], np.int64)
    scores, x, y = oc.observations(ix, logits, targets)
    assert np.array_equal(scores, np.array([[0, 0.5, 0.5], [1, 1, np.nan], [0.5, np.nan, np.nan]],
                                           np.float32), equal_nan=True)
    assert x[0] == 0.25 and y[0] == 8.75
    assert x[1] == 0.0625 and y[1] == 15.9375
    assert math.isnan(x[2]) and math.isnan(y[2])
    # S_max: pair scores sorted 0, .5, .5, .5, 1, 1 (m = 6)
    t, pairs, queries = oc.fit_s_max(scores, 0.5)          # position 2
    assert t == 0.5 and pairs == 4 / 6 and queries == 2 / 3
    t, pairs, queries = oc.fit_s_max(scores, 1.0)          # position 5
    assert t == 1.0 and pairs == 1.0 and queries == 1.0
    t, _, queries = oc.fit_s_max(scores, 0.0)              # position 0
    assert t == 0.0 and queries == 0.0


X8 = np.array([0.1, 0.2, 0.3, 0.4, 0.5, 0.6, 0.7, 0.8], np.float32)


@pytest.mark.parametrize("x,y,bins,q,want", [
    # 2 bins of 4: points at sorted positions 1 and 5; quantile entries ceil(q m) - 1
    (X8, [3, 1, 2, 0, 5, 4, 7, 6], 2, 0.5, ((0.2, 0.6), (1, 5))),
    (X8, [3, 1, 2, 0, 5, 4, 7, 6], 2, 1.0, ((0.2, 0.6), (3, 7))),
    (X8, [3, 1, 2, 0, 5, 4, 7, 6], 2, 0.0, ((0.2, 0.6), (0, 4))),
    # decreasing quantiles: the running maximum flattens the curve
    (X8, [9, 9, 9, 9, 1, 1, 1, 1], 2, 0.5, ((0.2, 0.6), (9, 9))),
    # 3 bins of 8 -> positions [0, 2), [2, 5), [5, 8): medians at 0, 3, 6
    (X8, [1, 2, 3, 4, 5, 6, 7, 8], 3, 0.5, ((0.1, 0.4, 0.7), (1, 4, 7))),
    # more bins than observations: one point per observation
    (X8[:3], [2, 1, 3], 16, 0.95, ((0.1, 0.2, 0.3), (2, 2, 3))),
    # equal x merge, keeping the larger quantile
    (np.array([1, 1, 1, 1, 2, 2, 2, 2], np.float32), [5, 6, 7, 8, 1, 2, 3, 4], 4, 1.0,
     ((1, 2), (8, 8))),
    # one x: three one-row bins merge into (2, 3), the flat curve through it
    (np.array([2, 2, 2], np.float32), [1, 3, 2], 4, 0.5, None),
    # nan x are left out
    (np.array([np.nan, 0.5, np.nan, 1.5], np.float32), [np.nan, 1, np.nan, 2], 2, 0.5,
     ((0.5, 1.5), (1, 2))),
])
def test_fit_gate_hand_worked(x, y, bins, q, want):
    got = oc.fit_gate(np.asarray(x, np.float32), np.asarray(y, np.float32), bins, q)
    if want is None:
        assert got[0][0] == 2 and got[0][1] == np.nextafter(np.float32(2), np.float32(3))
        assert got[1] == (3, 3)
        return
    assert np.array_equal(np.array(got[0], np.float32), np.array(want[0], np.float32))
    assert np.array_equal(np.array(got[1], np.float32), np.array(want[1], np.float32))


def test_fit_gate_empty_and_curve_is_valid():
    assert oc.fit_gate(np.array([np.nan], np.float32), np.array([np.nan], np.float32), 4, 0.9) is None
    rng = np.random.default_rng(5)
    for n in (1, 2, 7, 100, 1000):
        x = rng.gamma(2.0, 1.0, n).astype(np.float32)
        x[rng.random(n) < 0.2] = np.float32(1.0)          # ties
        y = (rng.gamma(1.5, 1.0, n) * (1 + x)).astype(np.float32)
        for bins in (1, 4, 16):
            xs, ys = oc.fit_gate(x, y, bins, 0.9)
            assert 2 <= len(xs) <= 16 and len(xs) == len(ys)
            assert all(a < c for a, c in zip(xs, xs[1:]))
            assert all(a <= c for a, c in zip(ys, ys[1:]))
            # every point is an observed x, or the one added to a single point
            seen = set(float(v) for v in x)
            assert all(float(v) in seen for v in xs) or (
                len(xs) == 2 and float(xs[0]) in seen and xs[1] == np.nextafter(xs[0], np.float32(np.inf)))
            p = oracle.params(gate_curve=(xs, ys))        # accepted as a curve
            assert p.gate_n == len(xs)

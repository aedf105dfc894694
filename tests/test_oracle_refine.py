"""Oracle refinement: exact squared L2 (uint8 as integers, Sec. 4.1.1) into a
top-k by (distance, id), with heap-quality early stopping counted in rounds
(Sec. 3.4.2, Algorithm 2's T_low rule, applied to refinement rounds).

The early-stop rule has no worked example in the paper, so it is pinned only
by hand-built candidate streams whose outcome follows from the rule's words."""
import numpy as np
import pytest

import oracle


def _u8(vals):
    return np.array(vals, np.uint8).reshape(-1, 1)


def test_stops_after_a_round_without_updates():
    q = np.array([100], np.uint8)
    rows = _u8([101, 103, 110, 120,   # round 1: top-2 becomes {0, 1}
                130, 140, 150, 160,   # round 2: no member changes -> low quality
                100, 99, 98, 97])     # round 3: would improve, never read
    ids = np.arange(12)
    p = oracle.params(round_size=4, t_low=1, u_min=1, f_min=1, r_min=1, alpha_front=0.5)
    out, d, st = oracle.refine_stream(q, rows, ids, 2, p)
    assert list(out) == [0, 1] and list(d) == [1.0, 9.0]
    assert list(st) == [8, 2]
    # early stop off: the whole stream is scored
    p0 = oracle.params(round_size=4, t_low=0)
    out, d, st = oracle.refine_stream(q, rows, ids, 2, p0)
    assert list(out) == [8, 0] and list(d) == [0.0, 1.0]  # d(id 9) = d(id 0) = 1: lower id
    assert list(st) == [12, 3]


def test_needs_consecutive_low_rounds_and_full_heap():
    q = np.array([0], np.uint8)
    rows = _u8([50, 60, 70, 80,  # r1: fills top-2 {0 (2500), 1 (3600)}
                90, 91, 92, 93,  # r2: low
                40, 95, 96, 97,  # r3: id 8 enters -> not low, counter resets
                98, 99, 99, 99,  # r4: low
                98, 99, 99, 99,  # r5: low -> stop with t_low = 2
                1, 1, 1, 1])     # r6: never read
    ids = np.arange(len(rows))
    p = oracle.params(round_size=4, t_low=2)
    out, d, st = oracle.refine_stream(q, rows, ids, 2, p)
    assert list(out) == [8, 0] and list(st) == [20, 5]
    # heap never full (k larger than the stream): no early stop at all
    out, d, st = oracle.refine_stream(q, rows, ids, 30, p)
    assert st[0] == len(rows) and list(out[:24]) == list(np.lexsort((ids, rows[:, 0])))
    assert list(out[24:]) == [-1] * 6 and np.all(np.isinf(d[24:]))


def test_r_min_delays_the_stop():
    q = np.array([0], np.uint8)
    rows = _u8([1, 2, 3, 4] + [200] * 12 + [0] * 4)
    ids = np.arange(len(rows))
    p = oracle.params(round_size=4, t_low=1, r_min=4)
    out, d, st = oracle.refine_stream(q, rows, ids, 2, p)
    assert list(st) == [16, 4] and list(out) == [0, 1]


def test_front_and_update_thresholds():
    # k = 4, alpha = 0.5 -> the front is the first 2 slots
    q = np.array([0], np.uint8)
    rows = _u8([10, 20, 30, 40,   # r1 fills
                35, 90, 90, 90])  # r2: one new member, in slot 3 (not front)
    ids = np.arange(8)
    base = dict(round_size=4, t_low=1, alpha_front=0.5, f_min=1)
    # u_min = 1: one update is enough -> not low -> no stop; stream ends after r2
    _, _, st = oracle.refine_stream(q, np.vstack([rows, _u8([95] * 4)]), np.arange(12), 4,
                                    oracle.params(u_min=1, **base))
    assert list(st) == [12, 3]
    # u_min = 2: 1 update < 2 and 0 front updates < 1 -> low -> stop after r2
    _, _, st = oracle.refine_stream(q, np.vstack([rows, _u8([95] * 4)]), np.arange(12), 4,
                                    oracle.params(u_min=2, **base))
    assert list(st) == [8, 2]
    # a front update alone keeps the round out of low quality
    rows2 = _u8([10, 20, 30, 40, 5, 90, 90, 90, 95, 95, 95, 95])
    _, _, st = oracle.refine_stream(q, rows2, np.arange(12), 4, oracle.params(u_min=2, **base))
    assert list(st) == [12, 3]


@pytest.mark.parametrize("dtype", ["u8", "f32"])
@pytest.mark.parametrize("k", [1, 10, 37])
def test_no_early_stop_equals_exact_topk(dtype, k):
    rng = np.random.default_rng(k)
    n, D = 1500, 24
    if dtype == "u8":
        rows = rng.integers(0, 8, size=(n, D)).astype(np.uint8)  # many exact ties
        q = rng.integers(0, 8, size=D).astype(np.uint8)
        dist = ((rows.astype(np.int64) - q.astype(np.int64)) ** 2).sum(1)
    else:
        rows = rng.standard_normal((n, D)).astype(np.float32)
        q = rng.standard_normal(D).astype(np.float32)
        dist = ((rows.astype(np.float64) - q.astype(np.float64)) ** 2).sum(1)
    ids = rng.permutation(n * 3)[:n]
    out, d, st = oracle.refine_stream(q, rows, ids, k, oracle.params(t_low=0, round_size=64))
    order = np.lexsort((ids, dist))[:k]
    if dtype == "u8":
        assert list(out) == list(ids[order]) and np.array_equal(d, dist[order].astype(np.float32))
    else:
        assert np.allclose(d, dist[order], rtol=1e-5)
        assert list(out) == list(ids[order])
    assert st[0] == n and st[1] == -(-n // 64)


def test_empty_stream_pads():
    out, d, st = oracle.refine_stream(np.zeros(4, np.uint8), np.zeros((0, 4), np.uint8),
                                      np.zeros(0, np.uint32), 3, oracle.params())
    assert list(out) == [-1, -1, -1] and np.all(np.isinf(d)) and list(st) == [0, 0]

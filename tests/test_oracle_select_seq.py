"""The sequential centroid stage of Algorithm 2 in the oracle: score bins
(Algorithm 1), centroid batches, the running d_min gate, a bounded heap of C
and the heap-quality stop. Pinned by a hand-worked index whose centroids make
every fp32 distance exact, and by the reduction to the order-independent
stage: one bin, one batch and no stop keep exactly the same clusters."""
import numpy as np
import pytest

import oracle
from nrix_writer import write_nrix


def hand_index(tmp_path):
    """b = 2, logit (0, 0), tau (0.5, 0.5): u0 = 0, both deviations 0.5, rank 0 =
    bit 0. Probe order {}, {r0}, {r1}, {r0, r1} -> codes 0, 1, 2, 3, scores 0,
    0.5, 0.5, 1.0; with S_max = 1 and 2 bins: bin 0 = {code 0}, bin 1 = the rest.
    code 0: clusters 0 (d 1), 1 (d 4); code 1: cluster 2 alone (d 9, C^dir);
    code 2: clusters 3 (d 0.25), 4 (d 9), 5 (d 0.25); code 3: clusters 6 (d 16),
    7 (d 1), 8 (d 2), 9 (d 0.0625)."""
    cent = np.array([[1, 0], [2, 0], [0, 3], [0.5, 0], [3, 0], [0, 0.5], [4, 0], [0, 1], [1, 1],
                     [0.25, 0]], np.float32)
    bkt = np.array([0, 2, 3, 6, 10], np.uint32)
    cl = np.arange(11, dtype=np.uint32)
    vec = np.zeros((10, 16), np.uint8)
    W = (np.zeros((4, 16), np.float32), np.zeros(4, np.float32), np.zeros((2, 4), np.float32),
         np.zeros(2, np.float32))
    path = str(tmp_path / "hand.nrix")
    write_nrix(path, vec, np.arange(10, dtype=np.uint32), bkt, cl, cent,
               np.array([0.5, 0.5], np.float32), *W)
    return oracle.Index(path)


def hand_probes():
    logit = np.zeros(2, np.float32)
    codes, keys, _ = oracle.probe_list(logit, np.array([0.5, 0.5], np.float32), 4, oracle.params())
    scores = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
    assert list(codes) == [0, 1, 2, 3] and list(scores) == [0.0, 0.5, 0.5, 1.0]
    return logit, codes, scores


BASE = dict(cent_mode=1, s_max=1.0, n_bins=2, b_batch=2, b_min=2, c_t_low=1, c_u_min=1, c_f_min=1,
            c_alpha_front=0.5, gate_m0=0.0, gate_m1=1.0)


# want_scored: centroid distances evaluated = the C^dir cluster 2 of bin 1 plus
# the clusters of the batches processed ([0, 1], [3, 4], [5, 6], [7, 8], then [9])
@pytest.mark.parametrize("kw,C,want_L,want_d,want_batches,want_scored", [
    # bin 0: batch [0, 1]: d_min 1, theta 2, H = {0}. bin 1: C^dir {2};
    # [3, 4]: d_min 0.25, theta 0.5 evicts 0, H = {3}; [5, 6]: H = {3, 5}, full;
    # [7, 8]: nothing within 0.5 -> low, t_low 1, H full, 2 bins -> stop before [9]
    (dict(), 2, [3, 5, 2], [0.25, 0.25, 9.0], 4, 1 + 8),
    # no early stop: [9]: d_min 0.0625, theta 0.125 evicts 3 and 5, H = {9}
    (dict(c_t_low=0), 2, [9, 2], [0.0625, 9.0], 5, 1 + 9),
    # B_min = 3 bins is never reached: no stop
    (dict(b_min=3), 2, [9, 2], [0.0625, 9.0], 5, 1 + 9),
    # C = 3: the heap is never full, no stop
    (dict(), 3, [9, 2], [0.0625, 9.0], 5, 1 + 9),
    # gate off: H keeps the C smallest of everything seen: (0.0625, 9), (0.25, 3)
    (dict(gate_m0=float("inf"), c_t_low=0), 2, [9, 3, 2], [0.0625, 0.25, 9.0], 5, 1 + 9),
])
def test_hand_worked_sequence(tmp_path, kw, C, want_L, want_d, want_batches, want_scored):
    ix = hand_index(tmp_path)
    logit, codes, scores = hand_probes()
    L, dL, ndir, nb, nsc = ix.cluster_list_seq(logit, codes, scores, C,
                                               oracle.params(**{**BASE, **kw}), with_scored=True)
    assert list(L) == want_L and list(dL) == want_d
    assert ndir == 1 and nb == want_batches and nsc == want_scored


def test_order_independent_stage_without_stop_equals_mode_0(tmp_path):
    """No stop, one bin, one batch: d_min is the global minimum, the gate is
    the final one, and the heap keeps the C smallest survivors; for m1 >= 0 the
    same holds with any bins and batches, since the running gate only
    tightens and an entry it evicts never returns."""
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, 20_000)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    path = str(tmp_path / "t.nrix")
    build_index(config(w.dtype, w.dim, w.hidden, 10, 8, 8), base, (W1, b1, W2[:10], b2[:10]), path)
    ix = oracle.Index(path)
    qs = synth.queries(w, 40)
    lg = ix.encode(qs)
    tau = ix.tau()
    for gate in ((float("inf"), 0.0), (0.0, 2.0), (0.5, 0.25)):
        for C in (4, 32, 400):
            p0 = oracle.params(gate_m0=gate[0], gate_m1=gate[1])
            for seq_kw in (dict(n_bins=1, b_batch=1 << 30), dict(n_bins=7, s_max=3.0, b_batch=5),
                           dict(n_bins=3, s_max=1.5, b_batch=1)):
                p1 = oracle.params(gate_m0=gate[0], gate_m1=gate[1], cent_mode=1, c_t_low=0, **seq_kw)
                for i in range(len(qs)):
                    codes, keys, _ = oracle.probe_list(lg[i], tau, 64, p1)
                    scores = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
                    L0, d0, n0 = ix.cluster_list(lg[i], codes, C, p0)
                    L1, d1, n1, _ = ix.cluster_list_seq(lg[i], codes, scores, C, p1)
                    assert np.array_equal(L0, L1) and np.array_equal(d0, d1) and n0 == n1


def test_search_uses_the_sequential_stage(tmp_path):
    """or_search with cent_mode 1 equals cluster_list_seq followed by the
    refinement of that list; with an early stop in narrow bins it keeps fewer
    clusters (the C^dir of bins never entered are left out)."""
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, 20_000)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    path = str(tmp_path / "t.nrix")
    build_index(config(w.dtype, w.dim, w.hidden, 10, 8, 8), base, (W1, b1, W2[:10], b2[:10]), path)
    ix = oracle.Index(path)
    qs = synth.queries(w, 30)
    kw = dict(cent_mode=1, n_bins=8, s_max=0.4, b_batch=4, b_min=1, c_t_low=1, gate_m0=0.0,
              gate_m1=4.0, t_low=0)
    ids, d, st = ix.search(qs, 10, 64, 4, oracle.params(**kw))
    ids0, d0, st0 = ix.search(qs, 10, 64, 4, oracle.params(**{**kw, "c_t_low": 0}))
    assert np.all(st[:, 2] <= st0[:, 2]) and np.any(st[:, 2] < st0[:, 2])
    lg = ix.encode(qs)
    tau = ix.tau()
    p = oracle.params(**kw)
    for i in range(len(qs)):
        codes, keys, _ = oracle.probe_list(lg[i], tau, 64, p)
        scores = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
        L, _, _, _ = ix.cluster_list_seq(lg[i], codes, scores, 4, p)
        assert st[i, 2] == len(L)


@pytest.mark.parametrize("curve,want", [
    # inside the curve: M(0.0625) = 0.5 + 0.0625 * 1 = 0.5625, theta 0.625: 9, 3, 5 pass
    (((0.0, 1.0), (0.5, 1.5)), [9, 3, 5, 2]),
    # d_min below the first point: M = y_0 = 0.25, theta 0.3125: 9, 3, 5 pass
    (((0.5, 1.0), (0.25, 2.0)), [9, 3, 5, 2]),
    # d_min past the last point: M = y_last = 1, theta 1.0625: 0 (d 1) and 7 (d 1) join
    (((0.01, 0.05), (1.0, 1.0)), [9, 3, 5, 0, 7, 2]),
    # three points, d_min on the second: segment 1, M = 0 + (0.0625 - 0.0625) s = 0,
    # theta 0.0625: only 9 passes
    (((0.0, 0.0625, 4.0), (0.0, 0.0, 8.0)), [9, 2]),
])
def test_calibrated_gate_curve(tmp_path, curve, want):
    """The piecewise-linear M of Sec. 3.4 on the hand-worked index (d_min over
    the non-singleton clusters = 0.0625): flat beyond its ends, linear inside,
    in both centroid stages."""
    ix = hand_index(tmp_path)
    logit, codes, scores = hand_probes()
    p0 = oracle.params(gate_curve=curve)
    L0, _, _ = ix.cluster_list(logit, codes, 8, p0)
    assert list(L0) == want
    p1 = oracle.params(gate_curve=curve, cent_mode=1, b_batch=1 << 20, c_t_low=0)
    L1, _, _, _ = ix.cluster_list_seq(logit, codes, scores, 8, p1)
    assert list(L1) == want


def test_gate_margin_closed_form_and_monotone():
    """M on dyadic breakpoints is the exact linear interpolation; an fp32 slope
    that rounds up (here (0.7287708 - 0.1917987) / (0.2216479 - 0.0459872))
    would put M one ulp above y_1 just left of x_1, so each segment is held
    within its end values; over random curves M never decreases, so the gate
    theta = x + M(x) does not either."""
    p = oracle.params(gate_curve=((0.0, 1.0, 3.0), (0.5, 1.0, 2.0)))
    for x, want in [(-1.0, 0.5), (0.0, 0.5), (0.25, 0.625), (1.0, 1.0), (2.0, 1.5), (2.5, 1.75),
                    (3.0, 2.0), (100.0, 2.0)]:
        assert oracle.gate_margin(p, x) == np.float32(want), x
    f = np.float32
    x0, x1, y0, y1 = f(0.04598718), f(0.22164789), f(0.19179872), f(0.72877085)
    p = oracle.params(gate_curve=((x0, x1), (y0, y1)))
    s = f(f(y1 - y0) / f(x1 - x0))
    just_left = np.nextafter(x1, f(0))
    assert f(np.float64(f(just_left - x0)) * np.float64(s) + np.float64(y0)) > y1  # would overshoot
    assert oracle.gate_margin(p, just_left) == y1
    rng = np.random.default_rng(9)
    for _ in range(200):
        n = int(rng.integers(2, 17))
        xs = np.sort(rng.choice(np.arange(1, 4000), n, replace=False)).astype(np.float32) * f(1e-4)
        ys = np.sort(rng.random(n).astype(np.float32))
        p = oracle.params(gate_curve=(xs, ys))
        probe = np.concatenate([xs, [np.nextafter(v, f(0)) for v in xs], [np.nextafter(v, f(1)) for v in xs],
                                rng.random(64).astype(np.float32) * f(0.5)])
        probe = np.sort(probe.astype(np.float32))
        m = np.array([oracle.gate_margin(p, v) for v in probe], np.float32)
        assert np.all(np.diff(m) >= 0)
        theta = (probe + m).astype(np.float32)
        assert np.all(np.diff(theta) >= 0)

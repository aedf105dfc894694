"""Calibration helpers on the GPU against the oracle: where rows are stored
(nr_index_locate) and centroid distances (nr_centroid_dists) bit for bit,
then the package's whole calibration (targets from a high-recall search,
scores, x, y, the fitted S_max and M) against the oracle's on the same
targets; the hand-worked index; argument checks."""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import build_small, need_cuda, recall
from oracle import calibrate as oc
from test_oracle_select_seq import hand_index

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return need_cuda()


@pytest.fixture(scope="module")
def tiny(torch, tmp_path_factory):
    from paper_2608_15438_gb300 import neuroute as nr

    path, base, _ = build_small(tmp_path_factory.mktemp("cal"), "tiny", n=100_000, bits=16)
    return {"ix": nr.Index(path, 0), "orc": oracle.Index(path), "base": base}


def test_locate_matches_oracle(tiny, torch):
    ix, orc = tiny["ix"], tiny["orc"]
    rng = np.random.default_rng(3)
    ids = np.concatenate([rng.integers(0, ix.N, 3000), rng.integers(0, 50, 200),   # repeats
                          [-5, ix.N, ix.N + 7, 1 << 40, 0, ix.N - 1]]).astype(np.int64)
    got = ix.locate(torch.from_numpy(ids).cuda()).cpu().numpy()
    want = np.array(oc.locate(orc, ids), np.int32)
    assert np.array_equal(got, want)
    everything = ix.locate(torch.arange(ix.N, device="cuda")).cpu().numpy()
    sizes = np.diff(orc.cl_off().astype(np.int64))
    assert np.array_equal(np.bincount(everything[:, 0], minlength=ix.n_clusters), sizes)
    assert ix.locate(torch.empty(0, dtype=torch.int64, device="cuda")).shape == (0, 4)


def test_centroid_dists_match_oracle(tiny, torch):
    ix, orc = tiny["ix"], tiny["orc"]
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 64)
    lg = orc.encode(qs)
    rng = np.random.default_rng(4)
    cl = rng.integers(0, ix.n_clusters, (64, 37)).astype(np.int32)
    cl[:, 0] = -1
    cl[:, 1] = ix.n_clusters
    d = ix.centroid_dists(torch.from_numpy(lg).cuda(), torch.from_numpy(cl).cuda()).cpu().numpy()
    for q in range(64):
        for j in range(37):
            assert d[q, j] == orc.centroid_dist(lg[q], int(cl[q, j])), (q, j)
    assert np.all(np.isinf(d[:, :2]))


def test_hand_worked_index(torch, tmp_path):
    from paper_2608_15438_gb300 import calibrate as pc
    from paper_2608_15438_gb300 import neuroute as nr

    hand_index(tmp_path)
    ix = nr.Index(str(tmp_path / "hand.nrix"), 0)
    tg = torch.tensor([[1, 2, 4], [9, 6, -1], [2, -1, -1]], dtype=torch.int64, device="cuda")
    assert ix.locate(tg[0]).cpu().tolist() == [[1, 0, 0, 2], [2, 1, 2, 1], [4, 2, 3, 3]]
    scores, x, y = pc.observations(ix, torch.zeros((3, 2), dtype=torch.float32, device="cuda"), tg)
    assert np.array_equal(scores, np.array([[0, 0.5, 0.5], [1, 1, np.nan], [0.5, np.nan, np.nan]],
                                           np.float32), equal_nan=True)
    assert x[0] == 0.25 and y[0] == 8.75 and x[1] == 0.0625 and y[1] == 15.9375
    assert np.isnan(x[2]) and np.isnan(y[2])
    ix.close()


def test_calibration_matches_oracle(tiny, torch):
    from paper_2608_15438_gb300 import calibrate as pc

    ix, orc = tiny["ix"], tiny["orc"]
    w = synth.WORKLOADS["tiny"]
    cq = synth.calib_queries(w, 300)
    dq = torch.from_numpy(cq).cuda()
    res = pc.calibrate(ix, dq, k=10, P=256, C=512, n_bins=8, quantile=0.9, coverage=0.95)
    lg = ix.encode(dq)
    targets = pc.targets_high_recall(ix, dq, lg, 10, 256, 512)
    truth = oracle.bruteforce(tiny["base"], cq, 10)[0]
    assert recall(targets.cpu().numpy(), truth) > 0.95       # the targets are the true neighbours
    scores, x, y = oc.observations(orc, lg.cpu().numpy(), targets.cpu().numpy())
    assert np.array_equal(res["scores"], scores, equal_nan=True)
    assert np.array_equal(res["x"], x, equal_nan=True) and np.array_equal(res["y"], y, equal_nan=True)
    assert res["n_gated"] > 250
    xs, ys = oc.fit_gate(x, y, 8, 0.9)
    assert np.array_equal(np.array(res["gate_curve"][0], np.float32), np.array(xs, np.float32))
    assert np.array_equal(np.array(res["gate_curve"][1], np.float32), np.array(ys, np.float32))
    assert (res["s_max"], res["pair_coverage"], res["query_coverage"]) == oc.fit_s_max(scores, 0.95)
    # the whole calibration in one library call (nr_calibrate) writes the same
    # curve and cutoff into the search parameters
    import ctypes

    from paper_2608_15438_gb300 import neuroute as nr

    p = nr.params(t_low=7)
    info = np.zeros(3, np.float64)
    assert nr.lib().nr_calibrate(ix.h, nr._ptr(lg), nr._ptr(targets), lg.shape[0], 10, 8, 0.9, 0.95,
                                 ctypes.byref(p), info.ctypes.data, nr._stream(None)) == 0
    assert p.gate_n == len(xs) and p.t_low == 7
    assert np.array_equal(np.array(p.gate_x[:p.gate_n], np.float32), np.array(xs, np.float32))
    assert np.array_equal(np.array(p.gate_y[:p.gate_n], np.float32), np.array(ys, np.float32))
    s_o, pc_o, qc_o = oc.fit_s_max(scores, 0.95)
    assert np.float32(p.s_max) == s_o and info[0] == pc_o and info[1] == qc_o
    assert info[2] == res["n_gated"]
    # the fitted curve is a valid gate and keeps the search near the targets
    ix.set_params(gate_curve=res["gate_curve"], t_low=0)
    try:
        ids, _ = ix.search_logits(dq, lg, 10, 256, 512)
    finally:
        ix.set_params()
    assert recall(ids.cpu().numpy(), targets.cpu().numpy()) > 0.8


def test_argument_checks(tiny, torch):
    from paper_2608_15438_gb300 import neuroute as nr

    ix = tiny["ix"]
    lib = nr.lib()
    import ctypes

    out = torch.empty((4, 4), dtype=torch.int32, device="cuda")
    ids = torch.zeros(4, dtype=torch.int64, device="cuda")
    assert lib.nr_index_locate(ix.h, ctypes.c_void_p(ids.data_ptr()), -1,
                               ctypes.c_void_p(out.data_ptr()), None) == -1
    assert lib.nr_index_locate(ix.h, None, 4, ctypes.c_void_p(out.data_ptr()), None) == -1
    lg = torch.zeros((2, ix.b), dtype=torch.float32, device="cuda")
    cl = torch.zeros((2, 3), dtype=torch.int32, device="cuda")
    assert lib.nr_centroid_dists(ix.h, ctypes.c_void_p(lg.data_ptr()), 2, ctypes.c_void_p(cl.data_ptr()),
                                 -1, None, None) == -1
    assert lib.nr_centroid_dists(ix.h, ctypes.c_void_p(lg.data_ptr()), 2, None, 3, None, None) == -1


@pytest.mark.parametrize("b", [2, 8, 16, 24])
def test_bucket_scores_match_oracle(torch, b):
    rng = np.random.default_rng(b)
    nq, k = 40, 12
    # dyadic logits on a coarse grid: many equal deviations and logits on tau
    logits = (rng.integers(-8, 9, (nq, b)) / 4).astype(np.float32)
    tau = (rng.integers(-2, 3, b) / 4).astype(np.float32)
    if b >= 8:
        logits[: nq // 2] = rng.normal(0, 1, (nq // 2, b)).astype(np.float32)
    codes = rng.integers(0, 1 << b, (nq, k)).astype(np.int64)
    codes[rng.random((nq, k)) < 0.1] = -1
    from paper_2608_15438_gb300 import calibrate as pc

    got = pc.bucket_scores(logits, tau, codes)
    for q in range(nq):
        for t in range(k):
            if codes[q, t] < 0:
                assert np.isnan(got[q, t])
            else:
                assert got[q, t] == oc.bucket_score(logits[q], tau, int(codes[q, t])), (q, t)

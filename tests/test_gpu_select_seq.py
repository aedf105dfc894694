"""The sequential centroid stage of Algorithm 2 on the GPU (cent_mode 1)
against the oracle: cluster lists and whole searches bit for bit, over score
bins, batch sizes, early stops and gates; the hand-worked index of the
oracle's pins; the reduction to the order-independent stage; argument
checks."""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import build_small, need_cuda
from test_oracle_select_seq import BASE, hand_index

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return need_cuda()


@pytest.fixture(scope="module")
def tiny(torch, tmp_path_factory):
    from paper_2608_15438_gb300 import neuroute as nr

    path, base, _ = build_small(tmp_path_factory.mktemp("seq"), "tiny", n=100_000, bits=16)
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 200)
    orc = oracle.Index(path)
    lg = orc.encode(qs)
    return {"ix": nr.Index(path, 0), "orc": orc, "q": qs, "lg": lg,
            "dq": torch.from_numpy(qs).cuda(), "dl": torch.from_numpy(lg).cuda()}


def oracle_lists(orc, lg, P, C, p):
    tau = orc.tau()
    out = []
    for i in range(len(lg)):
        codes, keys, _ = oracle.probe_list(lg[i], tau, P, p)
        scores = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
        out.append(orc.cluster_list_seq(lg[i], codes, scores, C, p)[0])
    return out


def test_hand_worked_index(torch, tmp_path):
    """The oracle's hand-worked sequence on the GPU (one query, logit (0, 0))."""
    from paper_2608_15438_gb300 import neuroute as nr

    hand_index(tmp_path)
    ix = nr.Index(str(tmp_path / "hand.nrix"), 0)
    dl = torch.zeros((1, 2), dtype=torch.float32, device="cuda")
    for kw, C, want in [(dict(), 2, [3, 5, 2]), (dict(c_t_low=0), 2, [9, 2]), (dict(b_min=3), 2, [9, 2]),
                        (dict(), 3, [9, 2]), (dict(gate_m0=float("inf"), c_t_low=0), 2, [9, 3, 2])]:
        ix.set_params(**{**BASE, **kw})
        cl, ncl = ix.debug_clusters(dl, 4, C)
        torch.cuda.synchronize()
        assert list(cl.cpu().numpy()[0, : int(ncl.item())]) == want, kw
    ix.close()


CASES = [
    dict(n_bins=1, b_batch=2048, c_t_low=0),                      # one bin, one batch, no stop
    dict(n_bins=8, s_max=0.6, b_batch=16, c_t_low=2, b_min=1),    # narrow bins, small batches
    dict(n_bins=4, s_max=1.0, b_batch=3, c_t_low=1, b_min=2, gate_m0=0.0, gate_m1=2.0),
    dict(n_bins=16, s_max=0.8, b_batch=64, c_t_low=1, c_u_min=2, c_f_min=1, c_alpha_front=0.7,
         gate_m0=0.0, gate_m1=4.0),
    dict(n_bins=2, s_max=2.0, b_batch=1, c_t_low=3, gate_m0=0.25, gate_m1=1.0),
    dict(n_bins=5, s_max=0.5, b_batch=7, c_t_low=1, gate_m0=3.0, gate_m1=-0.5),   # decreasing M
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
@pytest.mark.parametrize("P,C", [(16, 4), (128, 32), (512, 256)])
def test_cluster_lists_match_oracle(tiny, torch, case, P, C):
    ix, orc = tiny["ix"], tiny["orc"]
    kw = dict(cent_mode=1, **case)
    ix.set_params(**kw)
    try:
        cl, ncl = ix.debug_clusters(tiny["dl"], P, C)
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    want = oracle_lists(orc, tiny["lg"], P, C, oracle.params(**kw))
    for i, L in enumerate(want):
        assert ncl[i] == len(L), i
        assert np.array_equal(cl[i, : len(L)], L), i
        assert np.all(cl[i, len(L):] == -1)


@pytest.mark.parametrize("case", CASES[1:4], ids=["1", "2", "3"])
def test_search_matches_oracle(tiny, torch, case):
    ix, orc = tiny["ix"], tiny["orc"]
    kw = dict(cent_mode=1, t_low=4, **case)
    ix.set_params(**kw)
    try:
        ids, d = ix.search_logits(tiny["dq"], tiny["dl"], 10, 128, 64)
        st = ix.query_stats(len(tiny["q"]))
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    ids_o, d_o, st_o = orc.search(tiny["q"], 10, 128, 64, oracle.params(**kw), logits=tiny["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)


def test_without_stop_equals_order_independent_stage(tiny, torch):
    """No stop and m1 >= 0: the sequential stage keeps the clusters of the
    order-independent one, whatever the bins and batches."""
    ix = tiny["ix"]
    for seq in (dict(n_bins=1, b_batch=2048), dict(n_bins=7, s_max=0.9, b_batch=5)):
        for gate in (dict(), dict(gate_m0=0.0, gate_m1=2.0)):
            ix.set_params(**gate)
            cl0, n0 = ix.debug_clusters(tiny["dl"], 256, 128)
            ix.set_params(cent_mode=1, c_t_low=0, **seq, **gate)
            cl1, n1 = ix.debug_clusters(tiny["dl"], 256, 128)
            torch.cuda.synchronize()
            assert torch.equal(n0, n1) and torch.equal(cl0, cl1)
    ix.set_params()


@pytest.fixture(scope="module")
def many(torch, tmp_path_factory):
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, info = build_small(tmp_path_factory.mktemp("seqmc"), "tiny", n=20000, bits=8, k_max=16, t=4,
                                name="mc")
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 100)
    orc = oracle.Index(path)
    lg = orc.encode(qs)
    return {"ix": nr.Index(path, 0), "orc": orc, "lg": lg, "dl": torch.from_numpy(lg).cuda(), "info": info}


@pytest.mark.parametrize("C,case", [(64, dict(n_bins=4, s_max=2.0, b_batch=100, c_t_low=2)),
                                    (2048, dict(n_bins=3, s_max=3.0, b_batch=700, c_t_low=1,
                                                gate_m0=0.0, gate_m1=1.0)),
                                    (4096, dict(n_bins=1, b_batch=2048, c_t_low=0))])
def test_many_clusters_large_heaps(many, torch, C, case):
    """Up to 16 clusters a bucket, all 256 buckets probed: batches up to 2,048
    and heaps up to 4,096."""
    ix, orc = many["ix"], many["orc"]
    kw = dict(cent_mode=1, **case)
    ix.set_params(**kw)
    try:
        cl, ncl = ix.debug_clusters(many["dl"], 256, C)
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    want = oracle_lists(orc, many["lg"], 256, C, oracle.params(**kw))
    for i, L in enumerate(want):
        assert ncl[i] == len(L) and np.array_equal(cl[i, : len(L)], L), i


def test_argument_checks(tiny, torch):
    from paper_2608_15438_gb300 import neuroute as nr

    ix = tiny["ix"]
    for bad in (dict(cent_mode=2), dict(cent_mode=1, b_batch=0), dict(cent_mode=1, b_batch=4096),
                dict(cent_mode=1, n_bins=0), dict(cent_mode=1, c_alpha_front=1.5),
                dict(cent_mode=1, c_t_low=-1)):
        with pytest.raises(nr.NRError):
            ix.set_params(**bad)
    ix.set_params(cent_mode=1)
    with pytest.raises(nr.NRError):
        ix.search_logits(tiny["dq"], tiny["dl"], 10, 4096, 64)   # P > 2048 in mode 1
    ix.set_params()


CURVES = [((0.0, 2.0, 6.0, 20.0), (0.5, 2.0, 3.0, 3.5)),
          ((1.0, 3.0), (0.0, 4.0)),
          ((0.5, 1.0, 1.5, 2.0, 2.5, 3.0, 3.5, 4.0, 5.0, 6.0, 7.0, 8.0, 9.0, 10.0, 12.0, 14.0),
           (0.1, 0.2, 0.4, 0.8, 1.0, 1.2, 1.3, 1.4, 1.5, 1.6, 1.7, 1.8, 1.9, 2.0, 2.1, 2.2))]


@pytest.mark.parametrize("curve", CURVES, ids=["4pt", "2pt", "16pt"])
@pytest.mark.parametrize("mode", [0, 1])
def test_calibrated_gate_curve_matches_oracle(tiny, torch, curve, mode):
    ix, orc = tiny["ix"], tiny["orc"]
    kw = dict(gate_curve=curve, cent_mode=mode)
    if mode == 1:
        kw.update(n_bins=8, s_max=0.6, b_batch=16, c_t_low=2)
    ix.set_params(**kw)
    try:
        cl, ncl = ix.debug_clusters(tiny["dl"], 256, 128)
        ids, d = ix.search_logits(tiny["dq"], tiny["dl"], 10, 256, 128)
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    p = oracle.params(**kw)
    tau = orc.tau()
    for i in range(len(tiny["q"])):
        codes, keys, _ = oracle.probe_list(tiny["lg"][i], tau, 256, p)
        if mode == 1:
            scores = (keys >> np.uint64(32)).astype(np.uint32).view(np.float32)
            L = orc.cluster_list_seq(tiny["lg"][i], codes, scores, 128, p)[0]
        else:
            L = orc.cluster_list(tiny["lg"][i], codes, 128, p)[0]
        assert ncl[i] == len(L) and np.array_equal(cl[i, : len(L)], L), i
    ids_o, d_o, _ = orc.search(tiny["q"], 10, 256, 128, p, logits=tiny["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)


def test_gate_curve_argument_checks(tiny, torch):
    from paper_2608_15438_gb300 import neuroute as nr

    ix = tiny["ix"]
    for bad in (((1.0,), (1.0,)), ((1.0, 1.0), (0.0, 1.0)), ((1.0, 2.0), (1.0, 0.5)),
                ((0.0, float("inf")), (0.0, 1.0)), ((0.0, 1.0), (float("nan"), 1.0))):
        with pytest.raises(nr.NRError):
            ix.set_params(gate_curve=bad)
    ix.set_params()

"""GPU query path (through the C ABI) against the oracle, element by element.

Integer and index results must be bit-identical when the GPU is fed the
oracle's logits: probe codes (Algorithm 1), cluster lists (Algorithm 2's
centroid stage), top-k ids and uint8 distances; fp32 distances are compared
exactly too (both sides evaluate the same sequential fmaf chain), which is
stricter than the 1e-5 relative tolerance allowed for them. Encoder logits
are compared normwise within 1e-2 of the oracle's double-precision forward.
"""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import build_small, need_cuda, recall
from nrix_writer import write_nrix

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return need_cuda()


@pytest.fixture(scope="module")
def tiny(torch, tiny_index):
    from paper_2608_15438_gb300 import neuroute as nr

    ix = nr.Index(tiny_index["path"], 0)
    orc = oracle.Index(tiny_index["path"])
    qs = tiny_index["queries"]
    lg = orc.encode(qs)
    return {"ix": ix, "orc": orc, "q": qs, "lg": lg, "dq": torch.from_numpy(qs).cuda(),
            "dl": torch.from_numpy(lg).cuda(), "base": tiny_index["base"]}


@pytest.mark.parametrize("P", [1, 2, 8, 64, 500, 4096])
def test_route_codes_bit_exact(tiny, torch, P):
    codes, nprobe = tiny["ix"].route(tiny["dl"], P)
    codes = codes.cpu().numpy().view(np.uint32)
    nprobe = nprobe.cpu().numpy()
    tau = tiny["orc"].tau()
    p = oracle.params()
    for i in range(0, len(tiny["q"]), 7 if P >= 500 else 1):
        exp, _, _ = oracle.probe_list(tiny["lg"][i], tau, P, p)
        assert nprobe[i] == len(exp)
        assert np.array_equal(codes[i, : len(exp)], exp), i
        assert np.all(codes[i, len(exp):] == 0xFFFFFFFF)


@pytest.mark.parametrize("kw", [dict(l_sel=6), dict(r_max=2), dict(s_max=0.05),
                                dict(l_sel=9, r_max=3, s_max=0.2)])
def test_route_filters_bit_exact(tiny, torch, kw):
    ix = tiny["ix"]
    ix.set_params(**kw)
    try:
        codes, nprobe = ix.route(tiny["dl"], 300)
    finally:
        ix.set_params()
    codes = codes.cpu().numpy().view(np.uint32)
    tau = tiny["orc"].tau()
    p = oracle.params(**kw)
    for i in range(0, len(tiny["q"]), 3):
        exp, _, _ = oracle.probe_list(tiny["lg"][i], tau, 300, p)
        assert int(nprobe[i]) == len(exp)
        assert np.array_equal(codes[i, : len(exp)], exp)


@pytest.mark.parametrize("P", [2, 63, 64, 65, 128, 129, 256, 257, 512, 513, 777, 1024, 1025, 1536,
                               2047, 2048, 2049, 4095, 4096])
@pytest.mark.parametrize("kind", ["encoded", "ties"])
def test_route_threshold_enumeration_bit_exact(tiny, torch, P, kind):
    """Every probe budget takes the block-wide threshold enumeration (both
    sides of each multiple of the block's stride in the subtree capacity of 2P
    keys); logits on a grid of 1/8 around tau give deviations with many ties
    and zeros, whose subtrees often outgrow the capacity or crowd one cost
    bucket of the final ordering (the block then falls back to the heap)."""
    ix, orc = tiny["ix"], tiny["orc"]
    tau = orc.tau()
    lg = tiny["lg"][:200]
    if kind == "ties":
        rng = np.random.default_rng(P)
        lg = (tau[None, :] + rng.integers(-3, 4, lg.shape) / 8).astype(np.float32)
    codes, nprobe = ix.route(torch.from_numpy(lg).cuda(), P)
    codes = codes.cpu().numpy().view(np.uint32)
    nprobe = nprobe.cpu().numpy()
    p = oracle.params()
    for i in range(len(lg)):
        exp, _, _ = oracle.probe_list(lg[i], tau, P, p)
        assert nprobe[i] == len(exp), i
        assert np.array_equal(codes[i, : len(exp)], exp), i
        assert np.all(codes[i, len(exp):] == 0xFFFFFFFF)


@pytest.mark.parametrize("kw", [dict(s_max=0.0), dict(s_max=-1.0), dict(s_max=0.3), dict(l_sel=5),
                                dict(l_sel=11, s_max=0.5), dict(l_sel=1)])
@pytest.mark.parametrize("P", [64, 1024])
def test_route_threshold_filters_bit_exact(tiny, torch, kw, P):
    ix = tiny["ix"]
    ix.set_params(**kw)
    try:
        codes, nprobe = ix.route(tiny["dl"][:150], P)
    finally:
        ix.set_params()
    codes = codes.cpu().numpy().view(np.uint32)
    tau = tiny["orc"].tau()
    p = oracle.params(**kw)
    for i in range(150):
        exp, _, _ = oracle.probe_list(tiny["lg"][i], tau, P, p)
        assert int(nprobe[i]) == len(exp), i
        assert np.array_equal(codes[i, : len(exp)], exp), i


@pytest.mark.parametrize("P", [1, 2, 8, 100, 500, 1024, 2048, 4096])
@pytest.mark.parametrize("kw", [dict(), dict(s_max=0.3), dict(s_max=0.05), dict(l_sel=9, r_max=3),
                                dict(l_sel=6), "ties"])
def test_route_nonempty_budget_bit_exact(tiny, torch, P, kw):
    """The non-empty budget (D3 variant) skips empty buckets without spending
    the budget, examining at most 4 P flip sets (the tiny index has many
    empty buckets, so the block's first enumeration of 2 P sets often holds
    too few non-empty ones and the heap continues; small S_max and L_sel
    exhaust the admissible sets first; tied deviations crowd cost buckets)."""
    ix, orc = tiny["ix"], tiny["orc"]
    lg = tiny["lg"][:100]
    if kw == "ties":
        rng = np.random.default_rng(P)
        tau = orc.tau()
        lg = (tau[None, :] + rng.integers(-3, 4, lg.shape) / 8).astype(np.float32)
        kw = dict()
    ix.set_params(nonempty_budget=1, **kw)
    try:
        codes, nprobe = ix.route(torch.from_numpy(lg).cuda(), P)
    finally:
        ix.set_params()
    codes = codes.cpu().numpy().view(np.uint32)
    nprobe = nprobe.cpu().numpy()
    p = oracle.params(nonempty_budget=1, **kw)
    bkt = orc.bkt_off()
    for i in range(100):
        exp, _ = orc.probe_list(lg[i], P, p)
        assert nprobe[i] == len(exp), i
        assert np.array_equal(codes[i, : len(exp)], exp), i
        assert np.all(codes[i, len(exp):] == 0xFFFFFFFF)
        assert np.all(bkt[exp.astype(np.int64) + 1] > bkt[exp])


@pytest.mark.parametrize("kw", [dict(t_low=4), dict(t_low=0, gate_m0=0.0, gate_m1=2.0),
                                dict(t_low=4, cent_mode=1, n_bins=4, s_max=1.0, c_t_low=2)])
def test_search_nonempty_budget_bit_exact(tiny, torch, kw):
    ix, orc = tiny["ix"], tiny["orc"]
    ix.set_params(nonempty_budget=1, **kw)
    try:
        ids, d = ix.search_logits(tiny["dq"], tiny["dl"], 10, 64, 128)
        st = ix.query_stats(len(tiny["q"]))
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    ids_o, d_o, st_o = orc.search(tiny["q"], 10, 64, 128, oracle.params(nonempty_budget=1, **kw),
                                  logits=tiny["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)


def test_route_b4_hand_order(torch, tmp_path):
    from paper_2608_15438_gb300 import neuroute as nr

    # a 4-bit index whose only purpose is to carry tau = 0 (vectors unused)
    bkt = np.zeros(17, np.uint32)
    bkt[1:] = 1
    path = str(tmp_path / "b4.nrix")
    write_nrix(path, np.zeros((1, 16), np.uint8), [0], bkt, [0, 1], np.zeros((1, 4)), np.zeros(4),
               np.zeros((2, 16)), np.zeros(2), np.zeros((4, 2)), np.zeros(4))
    ix = nr.Index(path, 0)
    lg = torch.tensor([[0.375, -0.125, 0.5, -0.25]], dtype=torch.float32, device="cuda")
    codes, n = ix.route(lg, 16)
    assert [f"{c:X}" for c in codes.cpu().numpy().view(np.uint32)[0]] == list("57D4F16C39E0B28A")


@pytest.mark.parametrize("P,C", [(1, 1), (8, 32), (64, 16), (256, 1000), (1024, 4096)])
@pytest.mark.parametrize("gate", [(float("inf"), 0.0), (2.0, 0.5), (0.0, 0.0), (0.0, 4.0),
                                  (3.0, -0.5), (-0.5, 1.0), (float("-inf"), 1.0)])
def test_cluster_list_bit_exact(tiny, torch, P, C, gate):
    """Gates: off, affine, zero-width, the 1e9 operating point's M(x) = 4x, a
    decreasing M (m1 < 0), a negative offset, and one that drops every
    non-singleton cluster."""
    ix, orc = tiny["ix"], tiny["orc"]
    ix.set_params(gate_m0=gate[0], gate_m1=gate[1])
    try:
        cl, ncl = ix.debug_clusters(tiny["dl"], P, C)
    finally:
        ix.set_params()
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    tau = orc.tau()
    p = oracle.params(gate_m0=gate[0], gate_m1=gate[1])
    for i in range(0, len(tiny["q"]), 5):
        codes, _, _ = oracle.probe_list(tiny["lg"][i], tau, P, p)
        L, _, _ = orc.cluster_list(tiny["lg"][i], codes, C, p)
        assert ncl[i] == len(L), i
        assert np.array_equal(cl[i, : len(L)], L), i
        assert np.all(cl[i, len(L):] == -1)


CASES = [dict(k=10, P=8, C=32), dict(k=10, P=128, C=256), dict(k=1, P=16, C=8),
         dict(k=100, P=64, C=64), dict(k=256, P=32, C=512), dict(k=10, P=512, C=2048, t_low=0),
         dict(k=10, P=64, C=128, round_size=32, t_low=1), dict(k=7, P=64, C=128, round_size=1024),
         dict(k=10, P=64, C=128, round_size=64, t_low=2, u_min=3, f_min=2, alpha_front=0.7, r_min=3),
         dict(k=10, P=64, C=64, gate_m0=1.0, gate_m1=0.25)]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
def test_search_logits_bit_exact_u8(tiny, torch, case):
    case = dict(case)
    k, P, C = case.pop("k"), case.pop("P"), case.pop("C")
    ix, orc = tiny["ix"], tiny["orc"]
    ix.set_params(**case)
    try:
        ids, d = ix.search_logits(tiny["dq"], tiny["dl"], k, P, C)
        st = ix.query_stats(len(tiny["q"]))
        torch.cuda.synchronize()
        tot = ix.last_stats()
    finally:
        ix.set_params()
    ids_o, d_o, st_o = orc.search(tiny["q"], k, P, C, oracle.params(**case), logits=tiny["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)
    assert tot.candidates == st_o[:, 0].sum() and tot.nq == len(tiny["q"])


@pytest.fixture(scope="module")
def f32small(torch, tmp_path_factory):
    from paper_2608_15438_gb300 import neuroute as nr

    path, base, info = build_small(tmp_path_factory.mktemp("f32"), "f32-10m", n=60000, bits=14,
                                   k_max=8, t=32, name="f32")
    w = synth.WORKLOADS["f32-10m"]
    qs = synth.queries(w, 500)
    orc = oracle.Index(path)
    lg = orc.encode(qs)
    return {"ix": nr.Index(path, 0), "orc": orc, "q": qs, "lg": lg, "base": base,
            "dq": torch.from_numpy(qs).cuda(), "dl": torch.from_numpy(lg).cuda()}


@pytest.mark.parametrize("k,P,C,extra", [(10, 8, 64, {}), (10, 32, 64, {}), (50, 128, 256, {"t_low": 0}),
                                         (10, 64, 64, {"round_size": 128, "t_low": 2})])
def test_search_logits_fp32(f32small, torch, k, P, C, extra):
    ix, orc = f32small["ix"], f32small["orc"]
    ix.set_params(**extra)
    try:
        ids, d = ix.search_logits(f32small["dq"], f32small["dl"], k, P, C)
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    ids_o, d_o, _ = orc.search(f32small["q"], k, P, C, oracle.params(**extra), logits=f32small["lg"])
    d = d.cpu().numpy()
    fin = np.isfinite(d_o)
    assert np.array_equal(np.isfinite(d), fin)
    assert np.all(np.abs(d[fin] - d_o[fin]) <= 1e-5 * np.abs(d_o[fin]))
    assert np.array_equal(ids.cpu().numpy(), ids_o)


def test_encoder_logits_within_tolerance(tiny, f32small, torch):
    for ctx in (tiny, f32small):
        lg = ctx["ix"].encode(ctx["dq"]).cpu().numpy().astype(np.float64)
        ref = ctx["lg"].astype(np.float64)
        err = np.abs(lg - ref).max(1)
        assert np.all(err <= 1e-2 * np.abs(ref).max(1))


def test_end_to_end_recall_matches_oracle(tiny, torch):
    from test_oracle_search import exact_knn

    ix, orc = tiny["ix"], tiny["orc"]
    gi, _ = exact_knn(tiny["base"], tiny["q"], 10)
    for P, C in [(8, 32), (64, 128)]:
        ids, _ = ix.search(tiny["dq"], 10, P, C)
        ids_o, _, _ = orc.search(tiny["q"], 10, P, C, oracle.params())
        r_g, r_o = recall(ids.cpu().numpy(), gi), recall(ids_o, gi)
        assert abs(r_g - r_o) <= 0.002, (P, C, r_g, r_o)


def test_host_buffers_equal_device_path(tiny, torch):
    ix = tiny["ix"]
    ids, d = ix.search(tiny["dq"], 10, 32, 64)
    hq = torch.from_numpy(tiny["q"]).pin_memory()
    hi, hd = ix.search_host(hq, 10, 32, 64)
    assert torch.equal(hi, ids.cpu()) and torch.equal(hd, d.cpu())


def test_empty_and_ragged_batches(tiny, torch):
    ix, orc = tiny["ix"], tiny["orc"]
    for nq in (0, 1, 3, 255, 257):
        ids, d = ix.search_logits(tiny["dq"][:nq], tiny["dl"][:nq], 10, 16, 32)
        ids_o, d_o, _ = orc.search(tiny["q"][:nq], 10, 16, 32, oracle.params(), logits=tiny["lg"][:nq])
        assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)


def test_more_k_than_candidates_pads(tiny, torch):
    ix, orc = tiny["ix"], tiny["orc"]
    ids, d = ix.search_logits(tiny["dq"][:50], tiny["dl"][:50], 256, 1, 1)
    ids_o, d_o, _ = orc.search(tiny["q"][:50], 256, 1, 1, oracle.params(), logits=tiny["lg"][:50])
    ids = ids.cpu().numpy()
    assert np.array_equal(ids, ids_o) and np.array_equal(d.cpu().numpy(), d_o)
    assert (ids == -1).any()


def test_invalid_arguments_are_rejected(tiny, torch):
    from paper_2608_15438_gb300 import neuroute as nr

    ix = tiny["ix"]
    for k, P, C in [(0, 8, 8), (257, 8, 8), (10, 0, 8), (10, 4097, 8), (10, 8, 0), (10, 8, 4097)]:
        with pytest.raises(nr.NRError) as e:
            ix.search(tiny["dq"][:4], k, P, C)
        assert e.value.status == -1
    with pytest.raises(nr.NRError):
        ix.set_params(round_size=100)
    with pytest.raises(nr.NRError):
        ix.set_params(alpha_front=1.5)


def test_malformed_files(torch, tmp_path):
    from paper_2608_15438_gb300 import neuroute as nr

    with pytest.raises(nr.NRError) as e:
        nr.Index(str(tmp_path / "missing.nrix"), 0)
    assert e.value.status == -2
    bkt = np.zeros(17, np.uint32)
    bkt[1:] = 1
    args = (np.zeros((1, 16), np.uint8), [0], bkt, [0, 1], np.zeros((1, 4)), np.zeros(4),
            np.zeros((2, 16)), np.zeros(2), np.zeros((4, 2)), np.zeros(4))
    path = str(tmp_path / "trunc.nrix")
    write_nrix(path, *args, truncate_to=300)
    with pytest.raises(nr.NRError) as e:
        nr.Index(path, 0)
    assert e.value.status == -3
    path = str(tmp_path / "rows.nrix")  # a 4-byte row is not a multiple of 16 bytes
    write_nrix(path, np.zeros((1, 4), np.uint8), *args[1:])
    with pytest.raises(nr.NRError) as e:
        nr.Index(path, 0)
    assert e.value.status == -3


def test_out_of_range_directory_is_flagged_not_faulted(torch, tmp_path):
    """bkt_off pointing past the cluster table and a reversed cl_off range are
    reported as NR_ERR_DEVICE_CHECK; the kernels skip the bad ranges."""
    from paper_2608_15438_gb300 import neuroute as nr

    b = 3
    bkt = np.array([0, 1, 3, 3, 9, 4, 4, 4, 4], np.uint32)  # code 3 -> [3, 9) past n_cl = 4
    cl_off = np.array([0, 2, 1, 4, 5], np.uint32)           # cluster 1 reversed
    vec = np.arange(5 * 16, dtype=np.uint8).reshape(5, 16)
    path = str(tmp_path / "bad.nrix")
    write_nrix(path, vec, np.arange(5), bkt, cl_off, np.zeros((4, b)), np.zeros(b),
               np.zeros((2, 16)), np.zeros(2), np.zeros((b, 2)), np.zeros(b), K_max=8)
    ix = nr.Index(path, 0)
    q = torch.zeros((4, 16), dtype=torch.uint8, device="cuda")
    lg = torch.tensor([[1, 1, -1], [-1, 1, -1], [1, -1, 1], [1, 1, 1]], dtype=torch.float32,
                      device="cuda")
    ids, d = ix.search_logits(q, lg, 5, 8, 8)
    torch.cuda.synchronize()
    with pytest.raises(nr.NRError) as e:
        ix.last_stats()
    assert e.value.status == -6
    assert ix.last_stats().nq == 4  # the flag is cleared once reported
    # the context is still usable and results are deterministic; clusters 0 and 2
    # overlap in this file, so row 1 (id 1) is scored twice
    ids2, _ = ix.search_logits(q, lg, 5, 8, 8)
    torch.cuda.synchronize()
    assert torch.equal(ids, ids2)
    assert ids.cpu().tolist()[0] == [0, 1, 1, 2, 3]


@pytest.fixture(scope="module")
def many_clusters(torch, tmp_path_factory):
    """b = 8 and up to 16 clusters per bucket: probing all 256 buckets gives
    about 4096 candidate clusters, more than select keeps in shared memory."""
    from paper_2608_15438_gb300 import neuroute as nr

    path, base, info = build_small(tmp_path_factory.mktemp("mc"), "tiny", n=20000, bits=8,
                                   k_max=16, t=4, name="mc")
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 300)
    orc = oracle.Index(path)
    lg = orc.encode(qs)
    return {"ix": nr.Index(path, 0), "orc": orc, "q": qs, "lg": lg, "info": info,
            "dq": torch.from_numpy(qs).cuda(), "dl": torch.from_numpy(lg).cuda()}


@pytest.mark.parametrize("C,m1", [(64, None), (4096, None), (64, 0.25), (4096, 0.25), (4096, 2.0),
                                  (4096, -0.5), (64, 40.0)])
def test_select_overflow_to_global_slab(many_clusters, torch, C, m1):
    """More candidate clusters than shared memory holds: sorted in the global
    slab (gate off), or, when the gate's survivors fit, moved back to shared
    memory before the sort."""
    mc = many_clusters
    assert mc["info"]["n_clusters"] > 2048
    ix, orc = mc["ix"], mc["orc"]
    kw = {} if m1 is None else dict(gate_m0=0.0, gate_m1=m1)
    ix.set_params(**kw)
    cl, ncl = ix.debug_clusters(mc["dl"], 256, C)
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    tau = orc.tau()
    p = oracle.params(**kw)
    for i in range(0, len(mc["q"]), 7):
        codes, _, _ = oracle.probe_list(mc["lg"][i], tau, 256, p)
        L, _, _ = orc.cluster_list(mc["lg"][i], codes, C, p)
        assert ncl[i] == len(L)
        assert np.array_equal(cl[i, : len(L)], L)
    ids, d = ix.search_logits(mc["dq"], mc["dl"], 10, 256, C)
    ids_o, d_o, _ = orc.search(mc["q"], 10, 256, C, p, logits=mc["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)


@pytest.mark.parametrize("C,m1", [(64, None), (4096, None), (64, 1.0)])
def test_select_overflow_tied_distances(torch, tmp_path, C, m1):
    """Every bucket of a 12-bit index holds 16 clusters with the same centroid,
    so the 65,536 candidate distances of an all-probing query tie: the
    overflow kernel's preselection cannot thin them out, and the list comes
    from the bitonic sort of the whole slab, ties broken by cluster index
    (and, with the gate on, every cluster sits exactly at d_min)."""
    from paper_2608_15438_gb300 import neuroute as nr

    b, K = 12, 16
    ncl = (1 << b) * K
    rng = np.random.default_rng(5)
    vec = rng.integers(0, 256, (ncl, 16)).astype(np.uint8)
    path = str(tmp_path / "tied.nrix")
    write_nrix(path, vec, np.arange(ncl), np.arange(0, ncl + 1, K), np.arange(ncl + 1),
               np.full((ncl, b), 0.25, np.float32), np.zeros(b), np.zeros((16, 16)), np.zeros(16),
               np.zeros((b, 16)), np.zeros(b), K_max=K)
    ix = nr.Index(path, 0)
    orc = oracle.Index(path)
    lg = rng.normal(0, 1, (4, b)).astype(np.float32)
    q = rng.integers(0, 256, (4, 16)).astype(np.uint8)
    kw = {} if m1 is None else dict(gate_m0=0.0, gate_m1=m1)
    ix.set_params(**kw)
    try:
        cl, ncl_q = ix.debug_clusters(torch.from_numpy(lg).cuda(), 1 << b, C)
        ids, d = ix.search_logits(torch.from_numpy(q).cuda(), torch.from_numpy(lg).cuda(), 10,
                                  1 << b, C)
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    p = oracle.params(**kw)
    cl, ncl_q = cl.cpu().numpy(), ncl_q.cpu().numpy()
    for i in range(4):
        codes, _, _ = oracle.probe_list(lg[i], orc.tau(), 1 << b, p)
        L, _, _ = orc.cluster_list(lg[i], codes, C, p)
        assert ncl_q[i] == len(L) == C and np.array_equal(cl[i, :C], L), i
    ids_o, d_o, _ = orc.search(q, 10, 1 << b, C, p, logits=lg)
    assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)
    ix.close()


@pytest.fixture(scope="module")
def wide(torch, tmp_path_factory):
    """b = 12, up to 16 clusters per bucket, so that P = 2048 and 4096 give
    probe_budget * K_max of 32,768 and 65,536 (the largest select sort)."""
    from paper_2608_15438_gb300 import neuroute as nr

    path, base, info = build_small(tmp_path_factory.mktemp("wide"), "tiny", n=40000, bits=12,
                                   k_max=16, t=2, name="wide")
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 64)
    orc = oracle.Index(path)
    lg = orc.encode(qs)
    return {"ix": nr.Index(path, 0), "orc": orc, "q": qs, "lg": lg, "info": info,
            "dq": torch.from_numpy(qs).cuda(), "dl": torch.from_numpy(lg).cuda()}


@pytest.mark.parametrize("P,C", [(2048, 4096), (4096, 1024)])
def test_select_largest_budgets(wide, torch, P, C):
    ix, orc = wide["ix"], wide["orc"]
    kw = dict(t_low=4, gate_m0=0.0, gate_m1=1.0)
    ix.set_params(**kw)
    try:
        cl, ncl = ix.debug_clusters(wide["dl"], P, C)
        ids, d = ix.search_logits(wide["dq"], wide["dl"], 10, P, C)
        st = ix.query_stats(len(wide["q"]))
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    cl, ncl = cl.cpu().numpy(), ncl.cpu().numpy()
    tau = orc.tau()
    p = oracle.params(**kw)
    for i in range(0, len(wide["q"]), 4):
        codes, _, _ = oracle.probe_list(wide["lg"][i], tau, P, p)
        L, _, _ = orc.cluster_list(wide["lg"][i], codes, C, p)
        assert ncl[i] == len(L) and np.array_equal(cl[i, : len(L)], L), i
    ids_o, d_o, st_o = orc.search(wide["q"], 10, P, C, p, logits=wide["lg"])
    assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)


@pytest.mark.parametrize("workload", ["tiny", "u8-10m", "f32-10m", "u8-1b"])
def test_encoder_large_batch(torch, tmp_path, workload):
    """Large batches (several 128-row tiles per SM, a ragged last tile) through
    the tensor-core encoder, for the four encoder shapes (H = 256, 512, 384,
    512; b = 16, 20, 20, 24)."""
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, _ = build_small(tmp_path, workload, n=20000, name="enc")
    w = synth.WORKLOADS[workload]
    x = synth.base(w, 60000)
    ix, orc = nr.Index(path, 0), oracle.Index(path)
    lg = ix.encode(torch.from_numpy(x).cuda()).cpu().numpy().astype(np.float64)
    ref = orc.encode(x).astype(np.float64)
    err = np.abs(lg - ref).max(1)
    assert np.all(err <= 1e-2 * np.abs(ref).max(1))
    assert np.median(err / np.abs(ref).max(1)) < 2e-3


@pytest.mark.parametrize("workload", ["tiny", "f32-10m"])
def test_encoder_tile_edges(torch, tmp_path, workload):
    """Tile edges of the persistent tensor-core encoder: one row, a partial
    tile, exactly one tile, one row past it, and two tiles per SM plus one row
    (one CTA's third tile holds a single row); the same batch twice gives the
    same bits; input rows that start 8 bytes past a 16-byte boundary take the
    CUDA-core kernel and agree within the same tolerance."""
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, _ = build_small(tmp_path, workload, n=20000, name="enc")
    w = synth.WORKLOADS[workload]
    n_max = 2 * torch.cuda.get_device_properties(0).multi_processor_count * 128 + 1
    x = synth.base(w, n_max)
    ix, orc = nr.Index(path, 0), oracle.Index(path)
    ref = orc.encode(x).astype(np.float64)
    dx = torch.from_numpy(x).cuda()

    def check(lg, n):
        lg = lg.cpu().numpy().astype(np.float64)
        assert lg.shape == (n, w.bits)
        err = np.abs(lg - ref[:n]).max(1)
        assert np.all(err <= 1e-2 * np.abs(ref[:n]).max(1))

    for n in (1, 127, 128, 129, n_max):
        check(ix.encode(dx[:n]), n)
    assert torch.equal(ix.encode(dx), ix.encode(dx))
    pad = 8 // dx.element_size()
    buf = torch.zeros(dx.numel() + pad, dtype=dx.dtype, device="cuda")
    shifted = buf[pad:].view(dx.shape)
    shifted.copy_(dx)
    assert shifted.data_ptr() % 16 == 8
    check(ix.encode(shifted), n_max)
    ix.close()


def test_encoder_wait_expiry_is_flagged_and_the_context_stays_usable(tiny, torch):
    """With wait_limit_us < 0 every hand-off wait of the tensor-core encoder
    that is not already complete when first tested expires: the kernel stops,
    drains its issued MMAs (under its own 1 s bound), frees its tensor memory
    and sets the device flag, which nr_last_stats reports as
    NR_ERR_DEVICE_CHECK and clears. With the default limit the next call
    encodes correctly on the same context."""
    from paper_2608_15438_gb300 import neuroute as nr

    ix = tiny["ix"]
    # the tensor-core kernel's shapes (D % 16 == 0, D <= 128, H % 128 == 0, b <= 32)
    assert ix.D % 16 == 0 and ix.D <= 128 and ix.H % 128 == 0 and ix.b <= 32
    ix.set_params(wait_limit_us=-1)
    try:
        ix.encode(tiny["dq"])
        torch.cuda.synchronize()
        with pytest.raises(nr.NRError) as e:
            ix.last_stats()
        assert e.value.status == -6  # NR_ERR_DEVICE_CHECK
    finally:
        ix.set_params()
    ix.last_stats()  # the flag was cleared
    lg = ix.encode(tiny["dq"]).cpu().numpy()
    ref = tiny["lg"]
    assert np.all(np.abs(lg - ref).max(1) <= 1e-2 * np.abs(ref).max(1))
    ix.last_stats()
    # a limit longer than any hand-off changes nothing
    ix.set_params(wait_limit_us=2_000_000)
    try:
        lg2 = ix.encode(tiny["dq"]).cpu().numpy()
        ix.last_stats()
    finally:
        ix.set_params()
    assert np.array_equal(lg2, lg)

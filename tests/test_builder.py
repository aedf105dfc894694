"""The host index builder (paper Sec. 3.3; thresholds Sec. 3.2.3) against what
its definition fixes: exact lower medians, codes, the two CSR levels, the
cluster-count rule, centroids that are the means of their members, rows in
(code, cluster, id) order, thread-count independence, and k-means on a hand-made
bucket whose two clusters are obvious."""
import os

import numpy as np
import pytest

import synth
from nrix_reader import read_nrix
from paper_2608_15438_gb300.builder import build_index, build_index_from_logits, config, encode


def small_case(n=20_000, b=10, K_max=4, t=16):
    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, n)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    weights = (W1, b1, W2[:b], b2[:b])
    cfg = config(w.dtype, w.dim, w.hidden, b, K_max, t)
    return cfg, base, weights


@pytest.fixture(scope="module")
def built(tmp_path_factory):
    cfg, base, weights = small_case()
    path = str(tmp_path_factory.mktemp("bld") / "a.nrix")
    info = build_index(cfg, base, weights, path)
    logits = encode(cfg, base, weights)
    return cfg, base, weights, logits, read_nrix(path), info, path


def codes_of(logits, tau):
    bits = (logits >= tau[None, :]).astype(np.uint64)
    return (bits << np.arange(logits.shape[1], dtype=np.uint64)[None, :]).sum(1).astype(np.int64)


def test_tau_is_exact_lower_median(built):
    _, _, _, logits, ix, _, _ = built
    n = logits.shape[0]
    for j in range(logits.shape[1]):
        col = np.sort(logits[:, j].astype(np.float64))
        assert ix["tau"][j] == np.float32(col[(n - 1) // 2])


def test_buckets_hold_their_code_and_rows_are_ordered(built):
    _, base, _, logits, ix, info, _ = built
    N, b = logits.shape
    ids = ix["ids"].astype(np.int64)
    assert np.array_equal(np.sort(ids), np.arange(N))           # a permutation
    assert np.array_equal(ix["vec"], base[ids])                 # rows follow ids
    code = codes_of(logits, ix["tau"])
    bkt, cl = ix["bkt_off"].astype(np.int64), ix["cl_off"].astype(np.int64)
    assert bkt[0] == 0 and bkt[-1] == ix["n_cl"] and np.all(np.diff(bkt) >= 0)
    assert cl[0] == 0 and cl[-1] == N and np.all(np.diff(cl) > 0)   # no empty cluster
    nonempty = np.nonzero(np.diff(bkt))[0]
    assert info["n_buckets"] == len(nonempty) and info["n_clusters"] == ix["n_cl"]
    counts = np.bincount(code, minlength=1 << b)
    assert np.array_equal(np.nonzero(counts)[0], nonempty)
    for u in nonempty:
        r0, r1 = cl[bkt[u]], cl[bkt[u + 1]]
        assert r1 - r0 == counts[u]
        assert np.all(code[ids[r0:r1]] == u)
        for c in range(bkt[u], bkt[u + 1]):                     # ids ascending in a cluster
            assert np.all(np.diff(ids[cl[c]:cl[c + 1]]) > 0)


def test_cluster_count_rule_and_means(built):
    cfg, _, _, logits, ix, info, _ = built
    ids = ix["ids"].astype(np.int64)
    bkt, cl = ix["bkt_off"].astype(np.int64), ix["cl_off"].astype(np.int64)
    single = 0
    for u in np.nonzero(np.diff(bkt))[0]:
        n = cl[bkt[u + 1]] - cl[bkt[u]]
        K = bkt[u + 1] - bkt[u]
        assert 1 <= K <= min(cfg.K_max, -(-n // cfg.t))
        single += K == 1
        for c in range(bkt[u], bkt[u + 1]):
            m = logits[ids[cl[c]:cl[c + 1]]].astype(np.float64).mean(0)
            assert np.allclose(ix["cent"][c], m, rtol=1e-6, atol=1e-6)
    assert info["single_cluster_buckets"] == single


def test_members_nearer_their_centroid_than_average(built):
    """Lloyd's rule: a bucket's rows are, on average, closer to their own
    centroid than to the bucket's other centroids."""
    _, _, _, logits, ix, _, _ = built
    ids = ix["ids"].astype(np.int64)
    bkt, cl = ix["bkt_off"].astype(np.int64), ix["cl_off"].astype(np.int64)
    own, other = [], []
    for u in np.nonzero(np.diff(bkt) >= 2)[0]:
        cents = ix["cent"][bkt[u]:bkt[u + 1]].astype(np.float64)
        for k, c in enumerate(range(bkt[u], bkt[u + 1])):
            x = logits[ids[cl[c]:cl[c + 1]]].astype(np.float64)
            d = ((x[:, None, :] - cents[None]) ** 2).sum(-1)
            own.append(d[:, k])
            other.append(np.delete(d, k, axis=1).min(1))
    own, other = np.concatenate(own), np.concatenate(other)
    assert len(own) > 1000
    assert np.mean(own <= other) > 0.9


def test_thread_count_does_not_change_the_file(built, tmp_path):
    cfg, base, weights, logits, _, _, path = built
    p1 = str(tmp_path / "t1.nrix")
    build_index_from_logits(cfg, base, logits, weights, p1, nthreads=1)
    p8 = str(tmp_path / "t8.nrix")
    build_index_from_logits(cfg, base, logits, weights, p8, nthreads=8)
    a, b8, ref = open(p1, "rb").read(), open(p8, "rb").read(), open(path, "rb").read()
    assert a == b8 == ref


def test_two_obvious_clusters(tmp_path):
    """b = 1, N = 401: the lower median is the smallest of the 201 high rows, so
    the upper bucket holds exactly the high rows: two tight groups (100 near 10,
    101 near 20) that k-means (K = ceil(201 / 101) = 2) must separate exactly."""
    rng = np.random.default_rng(0)
    n = 401
    lg = np.zeros((n, 1), np.float32)
    lg[:200, 0] = -5.0 + rng.uniform(-0.1, 0.1, 200).astype(np.float32)
    grp = rng.permutation(np.r_[np.zeros(100), np.ones(101)]).astype(bool)
    lg[200:, 0] = np.where(grp, 20.0, 10.0) + rng.uniform(-0.1, 0.1, 201).astype(np.float32)
    base = rng.integers(0, 256, (n, 16), dtype=np.uint8)
    W = (np.zeros((4, 16), np.float32), np.zeros(4, np.float32), np.zeros((1, 4), np.float32),
         np.zeros(1, np.float32))
    p = str(tmp_path / "two.nrix")
    build_index_from_logits(config("u8", 16, 4, 1, 4, 101), base, lg, W, p)
    ix = read_nrix(p)
    bkt, cl, ids = ix["bkt_off"], ix["cl_off"], ix["ids"].astype(np.int64)
    assert list(bkt) == [0, 2, 4]
    hi = {frozenset(ids[cl[c]:cl[c + 1]].tolist()) for c in (2, 3)}
    want = {frozenset((200 + np.nonzero(~grp)[0]).tolist()), frozenset((200 + np.nonzero(grp)[0]).tolist())}
    assert hi == want
    c = sorted(float(v) for v in ix["cent"][2:4, 0])
    assert abs(c[0] - 10.0) < 0.05 and abs(c[1] - 20.0) < 0.05


def test_median_in_total_order_of_bit_patterns(tmp_path):
    """-0.0 sorts below +0.0: the lower median of (-0, +0, +0) is +0, of
    (-0, -0, +0) is -0."""
    base = np.zeros((3, 16), np.uint8)
    W = (np.zeros((4, 16), np.float32), np.zeros(4, np.float32), np.zeros((1, 4), np.float32),
         np.zeros(1, np.float32))
    for col, want in (([-0.0, 0.0, 0.0], 0x00000000), ([-0.0, -0.0, 0.0], 0x80000000)):
        p = str(tmp_path / "z.nrix")
        build_index_from_logits(config("u8", 16, 4, 1, 1, 8), base,
                                np.array(col, np.float32)[:, None], W, p)
        assert read_nrix(p)["tau"].view(np.uint32)[0] == want


def test_rejects_non_finite_logits(tmp_path):
    base = np.zeros((4, 16), np.uint8)
    W = (np.zeros((4, 16), np.float32), np.zeros(4, np.float32), np.zeros((1, 4), np.float32),
         np.zeros(1, np.float32))
    for bad in (np.nan, np.inf):
        lg = np.array([[0.0], [1.0], [bad], [2.0]], np.float32)
        with pytest.raises(RuntimeError):
            build_index_from_logits(config("u8", 16, 4, 1, 1, 8), base, lg, W,
                                    str(tmp_path / "bad.nrix"))
    assert not os.path.exists(str(tmp_path / "bad.nrix"))

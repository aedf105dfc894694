"""The non-empty probe budget (the D3 variant): flip sets in key order whose
buckets hold no cluster are enumerated but not spent. Pinned on a hand index
with empty buckets (b = 2, probe order 0, 1, 2, 3 for logit (0, 0)), and by its
definition as the non-empty subsequence of the plain probe list of
NR_NONEMPTY_SCAN * P codes."""
import numpy as np
import pytest

import oracle
from nrix_writer import write_nrix


def index_with(tmp_path, bkt, b=2):
    """tau = 0.5 on every bit, one row per cluster; bkt = the directory."""
    ncl = bkt[-1]
    cent = np.zeros((ncl, b), np.float32)
    cent[:, 0] = np.arange(ncl, dtype=np.float32)
    vec = np.zeros((ncl, 16), np.uint8)
    W = (np.zeros((4, 16), np.float32), np.zeros(4, np.float32), np.zeros((b, 4), np.float32),
         np.zeros(b, np.float32))
    path = str(tmp_path / "ne.nrix")
    write_nrix(path, vec, np.arange(ncl, dtype=np.uint32), np.array(bkt, np.uint32),
               np.arange(ncl + 1, dtype=np.uint32), cent, np.full(b, 0.5, np.float32), *W)
    return oracle.Index(path)


@pytest.mark.parametrize("bkt,P,want", [
    ([0, 2, 2, 5, 9], 2, [0, 2]),          # code 1 empty: skipped, not counted
    ([0, 2, 2, 5, 9], 3, [0, 2, 3]),
    ([0, 2, 2, 5, 9], 4, [0, 2, 3]),       # only three buckets hold clusters
    ([0, 0, 3, 3, 4], 1, [1]),             # empty base bucket: the first non-empty code
    ([0, 0, 3, 3, 4], 2, [1, 3]),
    ([0, 0, 0, 0, 4], 1, [3]),             # the scan of 4 P = 4 flip sets covers all four codes
    ([0, 0, 0, 0, 4], 2, [3]),
])
def test_hand_index(tmp_path, bkt, P, want):
    ix = index_with(tmp_path, bkt)
    logit = np.zeros(2, np.float32)
    codes, keys = ix.probe_list(logit, P, oracle.params(nonempty_budget=1))
    assert list(codes) == want
    plain, _ = ix.probe_list(logit, 4, oracle.params())
    assert list(plain) == [0, 1, 2, 3]


def test_scan_limit(tmp_path):
    """b = 3, all deviations 0.5: probe order 0, 1, 2, 4, 3, 5, 6, 7 (cost,
    then size, then rank mask). Only code 7 holds a cluster: P = 1 examines 4
    flip sets and lists nothing; P = 2 examines all 8 and lists 7."""
    bkt = [0, 0, 0, 0, 0, 0, 0, 0, 1]
    ix = index_with(tmp_path, bkt, b=3)
    logit = np.zeros(3, np.float32)
    plain, _ = ix.probe_list(logit, 8, oracle.params())
    assert list(plain) == [0, 1, 2, 4, 3, 5, 6, 7]
    assert list(ix.probe_list(logit, 1, oracle.params(nonempty_budget=1))[0]) == []
    assert list(ix.probe_list(logit, 2, oracle.params(nonempty_budget=1))[0]) == [7]


def test_is_the_nonempty_subsequence(tmp_path):
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, 20_000)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    path = str(tmp_path / "t.nrix")
    build_index(config(w.dtype, w.dim, w.hidden, 12, 4, 8), base, (W1, b1, W2[:12], b2[:12]), path)
    ix = oracle.Index(path)
    bkt = ix.bkt_off()
    lg = ix.encode(synth.queries(w, 30))
    assert np.mean(bkt[1:] == bkt[:-1]) > 0.1    # the index has empty buckets
    for kw in (dict(), dict(s_max=0.5), dict(l_sel=7)):
        for P in (1, 16, 100):
            for i in range(len(lg)):
                got, gk = ix.probe_list(lg[i], P, oracle.params(nonempty_budget=1, **kw))
                plain, pk = ix.probe_list(lg[i], 4 * P, oracle.params(**kw))
                keep = bkt[plain.astype(np.int64) + 1] > bkt[plain]
                assert np.array_equal(got, plain[keep][:P])
                assert np.array_equal(gk, pk[keep][:P])
                assert len(got) == P or len(got) == int(keep.sum())

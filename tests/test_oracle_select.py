"""Oracle centroid stage (Sec. 3.4.2 and Algorithm 2: singleton buckets to
C^dir, centroid distances in logit space, gate theta = d_min + M(d_min),
top-C) on a hand-made index with dyadic values, so every fp32 operation is
exact and a plain float64 restatement must agree bit for bit."""
import numpy as np
import pytest

import oracle
from nrix_writer import write_nrix

B = 3
# clusters per code (8 codes): code 0 one cluster, code 1 three, code 2 none,
# code 3 two, code 4 one, code 5 four, code 6 none, code 7 two
PER_CODE = [1, 3, 0, 2, 1, 4, 0, 2]


def _hand_index(tmp_path):
    rng = np.random.default_rng(11)
    bkt = np.concatenate([[0], np.cumsum(PER_CODE)]).astype(np.uint32)
    n_cl = int(bkt[-1])
    sizes = rng.integers(1, 5, size=n_cl)
    cl_off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.uint32)
    N = int(cl_off[-1])
    cent = rng.integers(-8, 9, size=(n_cl, B)).astype(np.float32) / 4  # dyadic
    vec = rng.integers(0, 256, size=(N, 4)).astype(np.uint8)
    W1 = np.zeros((2, 4), np.float32)
    W2 = np.zeros((B, 2), np.float32)
    path = str(tmp_path / "hand.nrix")
    write_nrix(path, vec, np.arange(N), bkt, cl_off, cent, np.zeros(B), W1, np.zeros(2), W2,
               np.zeros(B))
    return oracle.Index(path), bkt, cent


def _expected(bkt, cent, logit, codes, C, m0, m1):
    d = ((cent.astype(np.float64) - logit.astype(np.float64)) ** 2).sum(1)
    direct, cand = [], []
    for u in codes:
        c0, c1 = int(bkt[u]), int(bkt[u + 1])
        if c1 - c0 == 1:
            direct.append(c0)
        else:
            cand.extend(range(c0, c1))
    if cand and np.isfinite(m0):
        dmin = min(d[c] for c in cand)
        theta = dmin + (m0 + m1 * dmin)
    else:
        theta = np.inf
    surv = sorted([c for c in cand if d[c] <= theta], key=lambda c: (d[c], c))[:C]
    return sorted(direct + surv, key=lambda c: (d[c], c)), d


@pytest.mark.parametrize("C", [1, 2, 3, 5, 100])
@pytest.mark.parametrize("gate", [(np.inf, 0.0), (0.5, 0.25), (0.0, 0.0), (2.0, 1.0)])
def test_cluster_list_matches_definition(tmp_path, C, gate):
    ix, bkt, cent = _hand_index(tmp_path)
    rng = np.random.default_rng(C)
    m0, m1 = gate
    p = oracle.params(gate_m0=m0, gate_m1=m1)
    for trial in range(10):
        logit = (rng.integers(-8, 9, size=B) / 4).astype(np.float32)
        codes = rng.permutation(8)[: rng.integers(1, 9)].astype(np.uint32)
        L, dL, ndir = ix.cluster_list(logit, codes, C, p)
        exp, d = _expected(bkt, cent, logit, codes, C, m0, m1)
        assert list(L) == exp
        assert np.array_equal(dL, d[exp].astype(np.float32))
        assert ndir == sum(1 for u in codes if PER_CODE[u] == 1)


def test_singletons_bypass_gate_and_budget(tmp_path):
    ix, bkt, cent = _hand_index(tmp_path)
    logit = np.array([5, 5, 5], np.float32)  # far from everything
    p = oracle.params(gate_m0=0.0, gate_m1=0.0)
    L, dL, ndir = ix.cluster_list(logit, np.array([0, 4, 1], np.uint32), 1, p)
    # both singleton clusters (codes 0 and 4) plus the single best of code 1
    assert ndir == 2 and len(L) == 3
    assert int(bkt[0]) in L and int(bkt[4]) in L

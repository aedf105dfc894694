"""Oracle probe order (Algorithm 1, bucket enumeration; Eq. 10 binarisation;
deviation scores of Sec. 3.2.3) pinned to a hand-enumerated b = 4 case and to
a brute-force sort of all 2^b flip sets."""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "probe_order_b4.txt")


def _golden():
    vals = {}
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        k, *rest = line.split()
        vals[k] = rest
    return (np.array(vals["logits"], np.float32), np.array(vals["tau"], np.float32),
            [int(c, 16) for c in vals["codes"]])


def test_b4_hand_enumerated_order():
    logits, tau, codes = _golden()
    got, keys, perm = oracle.probe_list(logits, tau, 16, oracle.params())
    assert list(perm) == [1, 3, 0, 2]
    assert list(got) == codes
    # prefixes: a budget P returns the first P codes
    for P in (1, 3, 5, 11):
        assert list(oracle.probe_list(logits, tau, P, oracle.params())[0]) == codes[:P]


def test_b4_costs_are_the_hand_sums():
    logits, tau, _ = _golden()
    _, keys, _ = oracle.probe_list(logits, tau, 16, oracle.params())
    costs = [oracle.unpack_key(k)[0] for k in keys]
    assert costs == [0, .125, .25, .375, .375, .5, .5, .625, .625, .75, .75, .875, .875, 1.0, 1.125, 1.25]


def _random_sd(rng, b, ties):
    if ties:
        sd = rng.integers(0, 4, size=b).astype(np.float32) * np.float32(0.25)
    else:
        sd = rng.random(b, dtype=np.float32)
    return sd


@pytest.mark.parametrize("b", [1, 2, 5, 9, 12, 16])
@pytest.mark.parametrize("ties", [False, True])
def test_best_first_equals_sort_of_all_subsets(b, ties):
    rng = np.random.default_rng(100 + b + 50 * ties)
    for trial in range(4):
        sd = _random_sd(rng, b, ties)
        P = int(rng.integers(1, min(1 << b, 3000) + 1))
        p = oracle.params()
        a = oracle.probe_order(sd, P, p)
        e = oracle.probe_order_allsubsets(sd, P, p)
        assert np.array_equal(a, e)
        assert len(a) == min(P, 1 << b)
        assert np.all(np.diff(a.astype(np.uint64)) > 0)  # keys strictly increase


@pytest.mark.parametrize("kw", [dict(l_sel=5), dict(r_max=2), dict(s_max=0.6),
                                dict(l_sel=7, r_max=3, s_max=1.1)])
def test_filters_match_all_subsets(kw):
    rng = np.random.default_rng(7)
    for _ in range(5):
        sd = _random_sd(rng, 12, False)
        p = oracle.params(**kw)
        a = oracle.probe_order(sd, 4096, p)
        e = oracle.probe_order_allsubsets(sd, 4096, p)
        assert np.array_equal(a, e)
        for key in a[1:]:
            cost, size, mask = oracle.unpack_key(key)
            if "l_sel" in kw:
                assert mask >> kw["l_sel"] == 0
            if "r_max" in kw:
                assert size <= kw["r_max"]
            if "s_max" in kw:
                assert cost <= kw["s_max"]


def test_probe_list_invariants():
    rng = np.random.default_rng(3)
    for b in (8, 16, 20, 24):
        for _ in range(3):
            logits = rng.standard_normal(b).astype(np.float32)
            tau = rng.standard_normal(b).astype(np.float32) * 0.1
            P = 300
            codes, keys, perm = oracle.probe_list(logits, tau, P, oracle.params())
            u0 = sum(1 << j for j in range(b) if logits[j] >= tau[j])
            assert codes[0] == u0
            assert len(set(codes.tolist())) == len(codes) == min(P, 1 << b)
            assert np.all(codes < (1 << b))
            delta = np.abs(logits - tau)
            assert np.array_equal(perm, np.lexsort((np.arange(b), delta)))
            for c, key in zip(codes, keys):
                _, size, rmask = oracle.unpack_key(key)
                flips = sum(1 << int(perm[r]) for r in range(b) if (rmask >> r) & 1)
                assert c == u0 ^ flips and bin(flips).count("1") == size


def test_zero_deviation_and_equal_logit_threshold():
    # l = tau sets the bit (Eq. 10 uses >=); a zero deviation still costs a flip in |F|
    logits = np.array([1.0, 0.5, -2.0], np.float32)
    tau = np.array([1.0, 0.0, 0.0], np.float32)
    codes, keys, perm = oracle.probe_list(logits, tau, 8, oracle.params())
    assert codes[0] == 0b011
    assert perm[0] == 0  # delta 0
    assert codes[1] == 0b010  # flip bit 0 at cost 0, after the base bucket
    assert oracle.unpack_key(keys[1])[:2] == (0.0, 1)

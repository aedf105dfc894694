"""Seeded input generator: Philox4x32-10 against its published known-answer
vectors (Salmon et al., SC'11; Random123 distribution), determinism, and the
shape of the synthetic workloads."""
import numpy as np

import synth


def test_philox_known_answers():
    # Random123 kat_vectors, philox4x32 with 10 rounds
    assert synth.philox4x32_10([0, 0, 0, 0], [0, 0]) == [0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8]
    assert synth.philox4x32_10([0xFFFFFFFF] * 4, [0xFFFFFFFF] * 2) == [
        0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD]
    assert synth.philox4x32_10([0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344],
                               [0xA4093822, 0x299F31D0]) == [0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1]


def test_rows_are_pure_functions_of_their_index():
    w = synth.WORKLOADS["tiny"]
    full = synth.mixture(w, synth.SEED_DATA, 0, 5000, nthreads=3)
    part = synth.mixture(w, synth.SEED_DATA, 1234, 777, nthreads=1)
    assert np.array_equal(full[1234:1234 + 777], part)
    again = synth.mixture(w, synth.SEED_DATA, 0, 5000, nthreads=7)
    assert np.array_equal(full, again)


def test_u8_mixture_statistics():
    w = synth.WORKLOADS["tiny"]
    x = synth.mixture(w, synth.SEED_DATA, 0, 20000).astype(np.float64)
    comp = synth.components(w, synth.SEED_DATA, 0, 20000)
    assert comp.min() >= 0 and comp.max() < w.mixture
    # every component drawn about equally often
    counts = np.bincount(comp, minlength=w.mixture)
    assert counts.min() > 20000 / w.mixture * 0.4
    # within-component spread is sigma (clipping is rare for centres in [20, 235])
    sel = comp == 7
    resid = x[sel] - x[sel].mean(0)
    assert abs(resid.std() - w.sigma) < 1.0
    assert x.min() >= 0 and x.max() <= 255


def test_f32_mixture_is_normalised():
    w = synth.WORKLOADS["f32-10m"]
    x = synth.mixture(w, synth.SEED_DATA, 0, 3000)
    assert x.dtype == np.float32 and x.shape == (3000, 96)
    assert np.allclose(np.linalg.norm(x.astype(np.float64), axis=1), 1.0, atol=1e-6)


def test_queries_differ_from_base_but_share_centres():
    w = synth.WORKLOADS["tiny"]
    b = synth.mixture(w, synth.SEED_DATA, 0, 100)
    q = synth.mixture(w, synth.SEED_QUERIES, 0, 100)
    assert not np.array_equal(b, q)
    # a query lies much closer to its nearest base row than to a random one
    xb = synth.base(w, 20000).astype(np.float64)
    d = ((xb[None, :, :] - q[:5, None, :].astype(np.float64)) ** 2).sum(-1)
    assert np.all(d.min(1) < 0.5 * np.median(d, 1))


def test_encoder_weights_scale():
    w = synth.WORKLOADS["tiny"]
    W1, b1, W2, b2 = synth.encoder_weights(w)
    assert W1.shape == (w.hidden, w.dim) and W2.shape == (w.bits, w.hidden)
    assert abs(W1.std() * np.sqrt(w.dim) - 1.0) < 0.02
    assert abs(W2.std() * np.sqrt(w.hidden) - 1.0) < 0.05
    assert not b1.any() and not b2.any()


def test_centres_are_the_rows_centres():
    """The exported centres are the ones the rows scatter around: the mean of
    a component's rows approaches its centre (u8: uniform in [20, 235])."""
    w = synth.WORKLOADS["tiny"]
    c = synth.centres(w)
    assert c.shape == (w.mixture, w.dim) and c.min() >= 20.0 and c.max() <= 235.0
    rows = synth.mixture(w, synth.SEED_DATA, 0, 20_000).astype(np.float64)
    comp = synth.components(w, synth.SEED_DATA, 0, 20_000)
    for m in range(3):
        sel = rows[comp == m]
        assert len(sel) > 30
        assert np.abs(sel.mean(0) - c[m]).max() < 5 * w.sigma / np.sqrt(len(sel)) + 1.0

"""Encoders with several hidden layers (the encoder table of the paper's
appendix: linear + ReLU hidden layers, a linear last layer), in the oracle,
the index file (version 2: the hidden layers after the first in an eleventh
section) and the host builder. Pinned by a hand-worked forward whose middle
layers both pass and cut values at the ReLU."""
import numpy as np
import pytest

import oracle
from nrix_reader import read_nrix
from nrix_writer import write_nrix

X = np.array([[1.0, 2.0]], np.float32)
W1 = np.array([[1, 0], [0, 1], [1, 1]], np.float32)     # h1 = relu(1, 2 - 1, 3 - 4) = (1, 1, 0)
B1 = np.array([0, -1, -4], np.float32)
M1 = (np.array([[1, -1, 5], [2, 1, 0]], np.float32), np.array([0.5, -2], np.float32))  # -> (0.5, 1)
W2 = np.array([[2], [-4]], np.float32)
B2 = np.array([1, 0], np.float32)


@pytest.mark.parametrize("m2,want", [
    ((np.array([[-1, 1]], np.float32), np.zeros(1, np.float32)), [2.0, -2.0]),   # h3 = 0.5
    ((np.array([[1, -1]], np.float32), np.zeros(1, np.float32)), [1.0, 0.0]),    # h3 = relu(-0.5) = 0
])
def test_hand_worked_forward(tmp_path, m2, want):
    weights = (W1, B1, W2, B2, (M1, m2))
    got = oracle.encode_weights(weights, 1.0, X)
    assert got.tolist() == [want]
    # the same encoder read from a version-2 index file
    path = str(tmp_path / "mlp.nrix")
    write_nrix(path, np.zeros((1, 4), np.float32), [0], [0, 1, 1, 1, 1], [0, 1], np.zeros((1, 2)),
               np.zeros(2), np.pad(W1, ((0, 0), (0, 2))), B1, W2, B2, mid=(M1, m2))
    ix = oracle.Index(path)
    assert ix.mid == (2, 1) and ix.H == 3
    assert ix.encode(np.pad(X, ((0, 0), (0, 2)))).tolist() == [want]


def test_single_hidden_layer_unchanged():
    rng = np.random.default_rng(0)
    w = (rng.normal(size=(8, 5)).astype(np.float32), rng.normal(size=8).astype(np.float32),
         rng.normal(size=(3, 8)).astype(np.float32), rng.normal(size=3).astype(np.float32))
    x = rng.normal(size=(4, 5)).astype(np.float32)
    assert np.array_equal(oracle.encode_weights(w, 1.0, x), oracle.encode_weights(w + ((),), 1.0, x))


def test_host_builder_writes_the_hidden_layers(tmp_path):
    import synth
    from paper_2608_15438_gb300.builder import build_index, config, encode

    rng = np.random.default_rng(1)
    D, widths, b = 48, (32, 24, 16), 10
    base = rng.normal(size=(3000, D)).astype(np.float32)
    base /= np.linalg.norm(base, axis=1, keepdims=True)
    W1 = (rng.normal(size=(widths[0], D)) / np.sqrt(D)).astype(np.float32)
    mid = tuple(((rng.normal(size=(w, p)) / np.sqrt(p)).astype(np.float32),
                 (0.01 * rng.normal(size=w)).astype(np.float32))
                for p, w in zip(widths[:-1], widths[1:]))
    W2 = (rng.normal(size=(b, widths[-1])) / np.sqrt(widths[-1])).astype(np.float32)
    weights = (W1, np.zeros(widths[0], np.float32), W2, np.zeros(b, np.float32), mid)
    cfg = config("f32", D, widths[0], b, 4, 8, mid=widths[1:])
    path = str(tmp_path / "m.nrix")
    build_index(cfg, base, weights, path)
    f = read_nrix(path)
    assert f["mid_w"] == list(widths[1:])
    assert np.array_equal(f["mid"], np.concatenate([np.concatenate([W.ravel(), bb]) for W, bb in mid]))
    assert np.array_equal(f["W2"], W2.ravel())
    # the builder's fp32 logits agree with the oracle's double forward, and
    # tau is their lower median
    lg = encode(cfg, base, weights)
    ref = oracle.encode_weights(weights, 1.0, base)
    assert np.max(np.abs(lg - ref)) <= 1e-5 * np.max(np.abs(ref))
    assert np.array_equal(f["tau"], np.sort(lg, axis=0)[(len(base) - 1) // 2])
    orc = oracle.Index(path)
    assert orc.mid == widths[1:]
    assert np.array_equal(orc.encode(base[:50]), ref[:50])

"""Oracle encoder (Sec. 3.2.1: l = E(x), one hidden ReLU layer; input scale
for uint8 data as in Sec. 4.1.1) against a closed form and a double GEMM."""
import numpy as np

import oracle
from nrix_writer import write_nrix


def _index_with(tmp_path, W1, W2, b1=None, b2=None, in_scale=1.0, D=None, b=None):
    H, D = W1.shape
    b = W2.shape[0]
    vec = np.zeros((1, D), np.uint8)
    path = str(tmp_path / "enc.nrix")
    bkt = np.zeros((1 << b) + 1, np.uint32)
    bkt[1:] = 1
    write_nrix(path, vec, [0], bkt, [0, 1], np.zeros((1, b)), np.zeros(b), W1,
               np.zeros(H) if b1 is None else b1, W2, np.zeros(b) if b2 is None else b2,
               in_scale=in_scale)
    return oracle.Index(path)


def test_closed_form_hand_weights(tmp_path):
    W1 = np.array([[1, 0, 0, 0], [0, -1, 0, 0], [0, 0, 1, 1]], np.float32)
    W2 = np.array([[1, 1, 0], [0, 0, 2]], np.float32)
    ix = _index_with(tmp_path, W1, W2, b1=np.array([0, 0, -1.5]), b2=np.array([0.25, 0]))
    x = np.array([[2, 3, 1, 5], [0, 0, 0, 0]], np.uint8)
    # h = relu([2, -3, 6 - 1.5]) = [2, 0, 4.5]; l = [2 + 0.25, 9]
    # h = relu([0, 0, -1.5]) = 0;               l = [0.25, 0]
    assert np.array_equal(ix.encode(x), np.array([[2.25, 9.0], [0.25, 0.0]], np.float32))


def test_input_scale_applies_before_the_first_layer(tmp_path):
    W1 = np.eye(2, dtype=np.float32)
    W2 = np.array([[1, -1]], np.float32)
    ix = _index_with(tmp_path, W1, W2, in_scale=0.5)
    x = np.array([[8, 2], [2, 8]], np.uint8)
    assert np.array_equal(ix.encode(x)[:, 0], np.array([3.0, -3.0], np.float32))


def test_matches_double_gemm(tmp_path):
    rng = np.random.default_rng(0)
    D, H, b = 128, 256, 16
    W1 = (rng.standard_normal((H, D)) / np.sqrt(D)).astype(np.float32)
    W2 = (rng.standard_normal((b, H)) / np.sqrt(H)).astype(np.float32)
    b1 = (rng.standard_normal(H) * 0.1).astype(np.float32)
    ix = _index_with(tmp_path, W1, W2, b1=b1, in_scale=1 / 255)
    x = rng.integers(0, 256, size=(50, D)).astype(np.uint8)
    s = np.float64(np.float32(1 / 255))
    h = np.maximum(0, (x.astype(np.float64) * s) @ W1.T.astype(np.float64) + b1)
    ref = h @ W2.T.astype(np.float64)
    got = ix.encode(x).astype(np.float64)
    # fp32 rounding of a double result: half an ulp
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0 ** -24 + 1e-30)


def test_encode_from_weights_equals_index_encode(tmp_path):
    """The index-free entry point runs the same forward pass as the index's."""
    from nrix_writer import write_nrix

    rng = np.random.default_rng(3)
    D, H, b = 16, 32, 6
    W1 = rng.normal(size=(H, D)).astype(np.float32)
    b1 = rng.normal(size=H).astype(np.float32)
    W2 = rng.normal(size=(b, H)).astype(np.float32)
    b2 = rng.normal(size=b).astype(np.float32)
    vec = rng.integers(0, 256, (40, D), dtype=np.uint8)
    path = str(tmp_path / "e.nrix")
    bkt = np.zeros((1 << b) + 1, np.uint32)
    bkt[1:] = 1
    write_nrix(path, vec, np.arange(40, dtype=np.uint32), bkt, np.array([0, 40], np.uint32),
               np.zeros((1, b), np.float32), np.zeros(b, np.float32), W1, b1, W2, b2,
               in_scale=1.0 / 255.0)
    ix = oracle.Index(path)
    want = ix.encode(vec)
    got = oracle.encode_weights((W1, b1, W2, b2), 1.0 / 255.0, vec)
    assert np.array_equal(got, want)

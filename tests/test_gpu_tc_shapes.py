"""Tensor-core encoder on shapes the benchmark workloads do not use, against
the oracle's double-precision forward, with nonzero biases (the seeded
encoders have none):

* uint8, D = 112, H = 640, b = 22: W1 and W2 leave room for one X tile only
  (the single-buffer hand-off), five hidden chunks, b % 4 != 0 (scalar logit
  stores), b = 22 as in the paper's 1e9 setting;
* uint8, D = 128, H = 128, b = 10: one hidden chunk per tile, layer 2 N = 16;
* fp32, D = 64, H = 256, b = 24: eight fp32 pieces per converter thread.

Each encodes a ragged batch of several tiles per SM, twice (same bits), and
once more into an output buffer that starts 4 bytes past a 16-byte boundary
(scalar stores)."""
import ctypes

import numpy as np
import pytest

import oracle
import synth
from gpu_util import need_cuda
from paper_2608_15438_gb300.builder import build_index, config

pytestmark = pytest.mark.gpu

SHAPES = [("u8", 112, 640, 22), ("u8", 128, 128, 10), ("f32", 64, 256, 24)]


def _weights(D, H, b, seed):
    rng = np.random.default_rng(seed)
    return (rng.normal(0, 1 / np.sqrt(D), (H, D)).astype(np.float32),
            rng.normal(0, 0.1, H).astype(np.float32),
            rng.normal(0, 1 / np.sqrt(H), (b, H)).astype(np.float32),
            rng.normal(0, 0.1, b).astype(np.float32))


def _rows(dtype, n, D, seed):
    rng = np.random.default_rng(seed)
    if dtype == "u8":
        return rng.integers(0, 256, (n, D), dtype=np.uint8)
    x = rng.normal(0, 1, (n, D)).astype(np.float32)
    return x / np.linalg.norm(x, axis=1, keepdims=True)


@pytest.mark.parametrize("dtype,D,H,b", SHAPES)
def test_encoder_shapes_with_biases(tmp_path, dtype, D, H, b):
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr

    W = _weights(D, H, b, D + H + b)
    path = str(tmp_path / "enc.nrix")
    build_index(config(dtype, D, H, b, 4, 32), _rows(dtype, 4000, D, 1), W, path)
    ix, orc = nr.Index(path, 0), oracle.Index(path)
    n = 2 * torch.cuda.get_device_properties(0).multi_processor_count * 128 + 77
    x = _rows(dtype, n, D, 2)
    ref = orc.encode(x).astype(np.float64)
    dx = torch.from_numpy(x).cuda()
    lg = ix.encode(dx)
    got = lg.cpu().numpy().astype(np.float64)
    err = np.abs(got - ref).max(1)
    assert np.all(err <= 1e-2 * np.abs(ref).max(1))
    assert torch.equal(ix.encode(dx), lg)
    # an output buffer 4 bytes past a 16-byte boundary
    buf = torch.full((n * b + 4,), float("nan"), dtype=torch.float32, device="cuda")
    st = nr.lib().nr_encode(ix.h, ctypes.c_void_p(dx.data_ptr()), n,
                            ctypes.c_void_p(buf.data_ptr() + 4),
                            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == nr.NR_OK
    assert torch.equal(buf[1:1 + n * b].view(n, b), lg)
    assert torch.isnan(buf[0]) and torch.isnan(buf[1 + n * b:]).all()
    ix.close()
    orc.close()

"""The Python binding checks every tensor it hands to the C ABI (dtype,
shape, row-major contiguity, the index's GPU or the host) and raises before
calling the library, so a wrong tensor never reaches a kernel as a bad
pointer. Runs without a GPU: the index object is made without loading a file
and the library is replaced by a stub that records any call."""
import numpy as np
import pytest
import torch

from paper_2608_15438_gb300 import neuroute as nr


class _Called(Exception):
    pass


@pytest.fixture
def ix(monkeypatch):
    def no_library():
        raise _Called()

    monkeypatch.setattr(nr, "lib", no_library)
    x = object.__new__(nr.Index)
    x.h, x.device = None, 0
    x.N, x.D, x.H, x.b, x.n_clusters, x.dtype_code, x.k_max, x.t = 1000, 16, 128, 4, 10, 0, 4, 32
    return x


def test_bad_tensors_are_rejected_before_the_library(ix):
    q = torch.zeros((8, 16), dtype=torch.uint8)
    ids = torch.zeros((8, 10), dtype=torch.int64)
    d = torch.zeros((8, 10), dtype=torch.float32)
    with pytest.raises(ValueError, match="cuda:0"):
        ix.search(q, 10, 8, 8)                                  # host tensor for a device call
    with pytest.raises(ValueError, match="cuda:0"):
        ix.encode(q)
    with pytest.raises(ValueError, match="dtype"):
        ix.route(torch.zeros((8, 4), dtype=torch.float64), 8)
    with pytest.raises(ValueError, match="dtype"):
        ix.search_host(q.float(), 10, 8, 8)                     # fp32 rows for a uint8 index
    with pytest.raises(ValueError, match="shape"):
        ix.search_host(torch.zeros((8, 17), dtype=torch.uint8), 10, 8, 8)
    with pytest.raises(ValueError, match="contiguous"):
        ix.search_host(torch.zeros((16, 8), dtype=torch.uint8).T, 10, 8, 8)
    with pytest.raises(ValueError, match="out ids"):
        ix.search_host(q, 10, 8, 8, out=(ids.int(), d))
    with pytest.raises(ValueError, match="out dists"):
        ix.search_host(q, 10, 8, 8, out=(ids, d[:4]))
    with pytest.raises(TypeError):
        ix.search_host(np.zeros((8, 16), np.uint8), 10, 8, 8)


def test_good_host_tensors_reach_the_library(ix):
    q = torch.zeros((8, 16), dtype=torch.uint8)
    with pytest.raises(_Called):
        ix.search_host(q, 10, 8, 8)
    with pytest.raises(_Called):
        ix.search_host(q, 10, 8, 8, out=(torch.zeros((8, 10), dtype=torch.int64),
                                         torch.zeros((8, 10), dtype=torch.float32)))
    ix.dtype_code = 1                                           # an fp32 index takes fp32 rows
    with pytest.raises(_Called):
        ix.search_host(q.float(), 10, 8, 8)

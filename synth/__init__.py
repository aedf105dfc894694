"""Seeded synthetic inputs shared by the oracle and the CUDA path.

Holds none of the search method's arithmetic: it draws Gaussian-mixture
vectors and N(0, 1/fan_in) encoder weights from the Philox4x32-10 generator
(Salmon et al., SC'11) implemented in ``synth.c``, and names the workloads.

The workloads stand in for the paper's BigANN (uint8, 128-d) and Deep1B
(fp32, 96-d) benchmarks (paper Sec. 4.1, Table "datasets_all"), which are not
available here: same dimensionality and value type, mixture-of-Gaussians
structure, sizes from 1e5 to 1e9.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None

# Philox keys of the four independent draws
SEED_DATA = 1
SEED_QUERIES = 2
SEED_ENCODER = 3
SEED_KMEANS = 4
SEED_CALIB = 5    # held-out calibration queries
STREAM_W1 = 1
STREAM_W2 = 2


def lib():
    global _LIB
    if _LIB is None:
        path = os.path.join(_HERE, "libsynth.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(path)
        L.synth_philox4x32_10.argtypes = [ctypes.POINTER(ctypes.c_uint32)] * 3
        L.synth_mixture.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int,
                                    ctypes.c_int, ctypes.c_double, ctypes.c_int64, ctypes.c_int64,
                                    ctypes.c_void_p, ctypes.c_int]
        L.synth_components.argtypes = [ctypes.c_uint64, ctypes.c_int, ctypes.c_int64,
                                       ctypes.c_int64, ctypes.c_void_p]
        L.synth_normal.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int64,
                                   ctypes.c_double, ctypes.c_void_p]
        L.synth_centres.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int,
                                    ctypes.c_void_p]
        _LIB = L
    return _LIB


_CUDA_LIB = None


def cuda_lib():
    """The GPU row generator (synth_cuda.cu)."""
    global _CUDA_LIB
    if _CUDA_LIB is None:
        path = os.path.join(_HERE, "libsynth_cuda.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(path)
        L.synth_mixture_cuda.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_double, ctypes.c_int64, ctypes.c_int64,
                                         ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        _CUDA_LIB = L
    return _CUDA_LIB


def philox4x32_10(ctr, key):
    c = (ctypes.c_uint32 * 4)(*ctr)
    k = (ctypes.c_uint32 * 2)(*key)
    o = (ctypes.c_uint32 * 4)()
    lib().synth_philox4x32_10(c, k, o)
    return [int(v) for v in o]


@dataclass(frozen=True)
class Workload:
    name: str
    n: int            # base vectors
    dim: int          # D
    dtype: str        # "u8" or "f32"
    mixture: int      # M components
    sigma: float
    nq: int           # queries
    hidden: int       # H
    bits: int         # b
    k_max: int        # centroids per bucket
    t: int            # target cluster capacity
    probe: tuple = (8,)
    clusters: tuple = (32,)
    k: int = 10
    notes: str = ""
    mid: tuple = ()   # encoder hidden widths after the first (H)

    @property
    def dtype_code(self) -> int:
        return 0 if self.dtype == "u8" else 1

    @property
    def row_bytes(self) -> int:
        return self.dim * (1 if self.dtype == "u8" else 4)

    @property
    def in_scale(self) -> float:
        return 1.0 / 255.0 if self.dtype == "u8" else 1.0


WORKLOADS = {
    # 1e5 uint8 x 128, 256 components: the small case the oracle finishes in seconds
    "tiny": Workload("tiny", 100_000, 128, "u8", 256, 18.0, 1000, 256, 16, 4, 32,
                     probe=(8,), clusters=(32,)),
    # 1e7 uint8 x 128, b = 20
    "u8-10m": Workload("u8-10m", 10_000_000, 128, "u8", 256, 18.0, 10_000, 512, 20, 8, 64,
                       probe=(4, 16, 64), clusters=(32, 128)),
    # 1e7 fp32 x 96, L2-normalised, b = 20
    "f32-10m": Workload("f32-10m", 10_000_000, 96, "f32", 1024, 0.3, 10_000, 384, 20, 8, 64,
                        probe=(8, 32), clusters=(64,)),
    # the 1e7 uint8 workload indexed without bucket-local clustering (one
    # cluster per bucket): the analogue of the paper's bucket-clustering ablation
    "u8-10m-nocl": Workload("u8-10m-nocl", 10_000_000, 128, "u8", 256, 18.0, 10_000, 512, 20, 1, 64,
                            probe=(64, 256), clusters=(256,)),
    # 3e7 uint8 x 128 with b = 19: the 1e9 workload's rows per code (~57) and
    # rows per component, small enough for full kernel profiles
    "u8-30m": Workload("u8-30m", 30_000_000, 128, "u8", 512, 18.0, 10_000, 512, 19, 16, 64),
    # 1e8 uint8 x 128, b = 24
    "u8-100m": Workload("u8-100m", 100_000_000, 128, "u8", 4096, 18.0, 10_000, 512, 24, 16, 64),
    # 1e9 uint8 x 128, b = 24
    "u8-1b": Workload("u8-1b", 1_000_000_000, 128, "u8", 16384, 18.0, 10_000, 512, 24, 16, 64),
    # 1e7 fp32 x 1536, L2-normalised, with the paper's high-dimensional encoder
    # shape 1536 -> 512 -> 256 -> 128 -> 64 -> 16 (four hidden layers), b = 16
    "f32-1536": Workload("f32-1536", 10_000_000, 1536, "f32", 1024, 0.3, 10_000, 512, 16, 16, 64,
                         mid=(256, 128, 64)),
    # the same at 1e6 rows (6 GB): small enough for full kernel profiles
    "f32-1536-1m": Workload("f32-1536-1m", 1_000_000, 1536, "f32", 1024, 0.3, 10_000, 512, 16, 16, 64,
                            mid=(256, 128, 64)),
}


def mixture(w: Workload, seed_rows: int, row0: int, n: int, nthreads: int | None = None,
            seed_centres: int = SEED_DATA) -> np.ndarray:
    """Rows [row0, row0+n) of the workload's mixture (centres from seed_centres)."""
    nthreads = nthreads or os.cpu_count() or 1
    out = np.empty((n, w.dim), dtype=np.uint8 if w.dtype == "u8" else np.float32)
    rc = lib().synth_mixture(w.dtype_code, seed_rows, seed_centres, w.mixture, w.dim, w.sigma,
                             row0, n, out.ctypes.data, nthreads)
    if rc != 0:
        raise RuntimeError("synth_mixture failed")
    return out


def base(w: Workload, n: int | None = None, nthreads: int | None = None) -> np.ndarray:
    return mixture(w, SEED_DATA, 0, w.n if n is None else n, nthreads)


def queries(w: Workload, nq: int | None = None, nthreads: int | None = None) -> np.ndarray:
    return mixture(w, SEED_QUERIES, 0, w.nq if nq is None else nq, nthreads)


def calib_queries(w: Workload, nq: int, nthreads: int | None = None) -> np.ndarray:
    """Held-out calibration queries: the query distribution on its own stream."""
    return mixture(w, SEED_CALIB, 0, nq, nthreads)


def components(w: Workload, seed_rows: int, row0: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    lib().synth_components(seed_rows, w.mixture, row0, n, out.ctypes.data)
    return out


def centres(w: Workload, seed_centres: int = SEED_DATA) -> np.ndarray:
    """The mixture centres [M x D] (float64) that the rows are drawn around."""
    out = np.empty((w.mixture, w.dim), np.float64)
    if lib().synth_centres(w.dtype_code, seed_centres, w.mixture, w.dim, out.ctypes.data) != 0:
        raise RuntimeError("synth_centres failed")
    return out


class DeviceRows:
    """Rows of a workload's mixture generated on a GPU (the definition of
    ``mixture``, computed by synth_cuda.cu), for bases too large for the host."""

    def __init__(self, w: Workload, seed_rows: int = SEED_DATA, seed_centres: int = SEED_DATA,
                 device: int = 0):
        import torch

        self.w, self.seed_rows, self.device = w, seed_rows, device
        self.cent = torch.from_numpy(centres(w, seed_centres)).to(f"cuda:{device}")

    def rows(self, row0: int, n: int, out=None, stream=None):
        """Rows [row0, row0 + n) as a CUDA tensor [n x D] (uint8 or float32)."""
        import torch

        w = self.w
        dt = torch.uint8 if w.dtype == "u8" else torch.float32
        if out is None:
            out = torch.empty((n, w.dim), dtype=dt, device=f"cuda:{self.device}")
        assert out.dtype == dt and out.is_contiguous() and out.shape[0] >= n
        s = stream if stream is not None else torch.cuda.current_stream(self.device)
        rc = cuda_lib().synth_mixture_cuda(w.dtype_code, self.seed_rows, w.mixture, w.dim, w.sigma,
                                           row0, n, ctypes.c_void_p(self.cent.data_ptr()),
                                           ctypes.c_void_p(out.data_ptr()),
                                           ctypes.c_void_p(s.cuda_stream))
        if rc != 0:
            raise RuntimeError("synth_mixture_cuda failed")
        return out[:n]


def normal(seed: int, stream: int, n: int, scale: float) -> np.ndarray:
    out = np.empty(n, dtype=np.float32)
    lib().synth_normal(seed, stream, n, scale, out.ctypes.data)
    return out


def encoder_weights(w: Workload, seed: int = SEED_ENCODER):
    """Seeded encoder D -> H (ReLU) [-> mid widths (ReLU)] -> b with
    N(0, 1/fan_in) weights, zero biases.

    Returns (W1 [H x D], b1 [H], W2 [b x H_last], b2 [b]) as fp32 arrays, and
    with hidden layers after the first a fifth element ((W, b), ...) of them
    (stream 3 + i for layer i)."""
    W1 = normal(seed, STREAM_W1, w.hidden * w.dim, 1.0 / np.sqrt(w.dim)).reshape(w.hidden, w.dim)
    widths = (w.hidden,) + tuple(w.mid)
    mid = tuple((normal(seed, 3 + i, wo * wi, 1.0 / np.sqrt(wi)).reshape(wo, wi), np.zeros(wo, np.float32))
                for i, (wi, wo) in enumerate(zip(widths[:-1], widths[1:])))
    hl = widths[-1]
    W2 = normal(seed, STREAM_W2, w.bits * hl, 1.0 / np.sqrt(hl)).reshape(w.bits, hl)
    out = (W1, np.zeros(w.hidden, np.float32), W2, np.zeros(w.bits, np.float32))
    return out + (mid,) if mid else out

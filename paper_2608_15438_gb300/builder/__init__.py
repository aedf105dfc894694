"""Index builder binding (``nrbuild.cpp``): a plain host routine run once, off
the query path, that writes the index file the query library loads.

Paper Sec. 3.3: encode the base, per-bit median thresholds (Sec. 3.2.3),
bucket by code, bucket-local k-means in logit space, CSR layout.

Encoder weights are (W1 [H x D], b1 [H], W2 [b x H_last], b2 [b]) fp32, with
an optional fifth element ((W [w x previous], b [w]), ...) holding the hidden
layers after the first (the encoder table of the paper's appendix: several
linear + ReLU layers, a linear last layer); H_last is the last hidden width.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None


class Config(ctypes.Structure):
    _fields_ = [("dtype", ctypes.c_int), ("D", ctypes.c_int), ("H", ctypes.c_int),
                ("b", ctypes.c_int), ("K_max", ctypes.c_int), ("t", ctypes.c_int),
                ("in_scale", ctypes.c_float), ("lloyd_iters", ctypes.c_int),
                ("sample_per_cluster", ctypes.c_int), ("seed", ctypes.c_uint64),
                ("n_mid", ctypes.c_int), ("mid_w", ctypes.c_int * 7)]


def lib():
    global _LIB
    if _LIB is None:
        path = os.path.join(_HERE, "libnrbuild.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(path)
        vp = ctypes.c_void_p
        L.nrb_build.argtypes = [ctypes.POINTER(Config), vp, ctypes.c_int64, vp, vp, vp, vp, vp,
                                ctypes.c_char_p, ctypes.c_int, vp]
        L.nrb_build.restype = ctypes.c_int
        L.nrb_build_logits.argtypes = [ctypes.POINTER(Config), vp, ctypes.c_int64, vp, vp, vp, vp,
                                       vp, vp, ctypes.c_char_p, ctypes.c_int, vp]
        L.nrb_build_logits.restype = ctypes.c_int
        L.nrb_encode.argtypes = [ctypes.POINTER(Config), vp, ctypes.c_int64, vp, vp, vp, vp, vp, vp,
                                 ctypes.c_int]
        L.nrb_encode.restype = ctypes.c_int
        _LIB = L
    return _LIB


def config(dtype: str, D: int, H: int, b: int, K_max: int, t: int, seed: int = 4,
           lloyd_iters: int = 5, sample_per_cluster: int = 256, mid=()) -> Config:
    """mid: widths of the hidden layers after the first (at most 7)."""
    if len(mid) > 7:
        raise ValueError("at most 7 hidden layers after the first")
    c = Config()
    c.dtype = 0 if dtype == "u8" else 1
    c.D, c.H, c.b, c.K_max, c.t = D, H, b, K_max, t
    c.in_scale = 1.0 / 255.0 if dtype == "u8" else 1.0
    c.lloyd_iters, c.sample_per_cluster, c.seed = lloyd_iters, sample_per_cluster, seed
    c.n_mid = len(mid)
    for i, v in enumerate(mid):
        c.mid_w[i] = int(v)
    return c


def split_weights(weights):
    """(W1, b1, W2, b2, Wm): fp32 contiguous arrays, Wm the middle layers'
    W then b concatenated as the file stores them (empty without any)."""
    W1, b1, W2, b2 = (np.ascontiguousarray(w, np.float32) for w in weights[:4])
    mid = weights[4] if len(weights) > 4 else ()
    parts = [np.concatenate([np.asarray(W, np.float32).ravel(), np.asarray(bb, np.float32).ravel()])
             for W, bb in mid]
    Wm = np.ascontiguousarray(np.concatenate(parts) if parts else np.zeros(1, np.float32))
    return W1, b1, W2, b2, Wm


def build_index(cfg: Config, base: np.ndarray, weights, path: str, nthreads: int | None = None):
    """Build the index over base [N x D] and write it to path. Returns a dict
    of index statistics."""
    base = np.ascontiguousarray(base)
    W1, b1, W2, b2, Wm = split_weights(weights)
    info = np.zeros(5, np.int64)
    rc = lib().nrb_build(ctypes.byref(cfg), base.ctypes.data, base.shape[0], W1.ctypes.data,
                         b1.ctypes.data, W2.ctypes.data, b2.ctypes.data, Wm.ctypes.data,
                         path.encode(), nthreads or os.cpu_count() or 1, info.ctypes.data)
    if rc != 0:
        raise RuntimeError(f"nrb_build failed ({rc})")
    return _info(info)


def _info(info):
    return {"n_clusters": int(info[0]), "n_buckets": int(info[1]), "max_bucket": int(info[2]),
            "max_cluster": int(info[3]), "single_cluster_buckets": int(info[4])}


def build_index_from_logits(cfg: Config, base: np.ndarray, logits: np.ndarray, weights, path: str,
                            nthreads: int | None = None):
    """Build the index over base [N x D] from given base logits [N x b] (the
    encoder step skipped) and write it to path. weights are stored in the file."""
    base = np.ascontiguousarray(base)
    logits = np.ascontiguousarray(logits, np.float32)
    if logits.shape != (base.shape[0], cfg.b):
        raise ValueError("logits must be [N x b]")
    W1, b1, W2, b2, Wm = split_weights(weights)
    info = np.zeros(5, np.int64)
    rc = lib().nrb_build_logits(ctypes.byref(cfg), base.ctypes.data, base.shape[0],
                                logits.ctypes.data, W1.ctypes.data, b1.ctypes.data, W2.ctypes.data,
                                b2.ctypes.data, Wm.ctypes.data, path.encode(),
                                nthreads or os.cpu_count() or 1, info.ctypes.data)
    if rc != 0:
        raise RuntimeError(f"nrb_build_logits failed ({rc})")
    return _info(info)


def encode(cfg: Config, base: np.ndarray, weights, nthreads: int | None = None) -> np.ndarray:
    """The builder's fp32 encoder over base [N x D]: logits [N x b]."""
    base = np.ascontiguousarray(base)
    W1, b1, W2, b2, Wm = split_weights(weights)
    out = np.empty((base.shape[0], cfg.b), np.float32)
    rc = lib().nrb_encode(ctypes.byref(cfg), base.ctypes.data, base.shape[0], W1.ctypes.data,
                          b1.ctypes.data, W2.ctypes.data, b2.ctypes.data, Wm.ctypes.data,
                          out.ctypes.data, nthreads or os.cpu_count() or 1)
    if rc != 0:
        raise RuntimeError(f"nrb_encode failed ({rc})")
    return out

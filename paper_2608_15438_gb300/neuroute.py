"""ctypes binding of libneuroute.so: the same entry points as
include/neuroute.h, argument marshalling only. Device buffers are torch CUDA
tensors (used for memory and streams only); every step of the search runs in
the library's kernels. There is no fallback: if the library is missing or a
call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libneuroute.so")
_LIB = None

NR_OK = 0
STATUS = {0: "NR_OK", -1: "NR_ERR_INVALID_ARG", -2: "NR_ERR_IO", -3: "NR_ERR_FORMAT",
          -4: "NR_ERR_OOM", -5: "NR_ERR_CUDA", -6: "NR_ERR_DEVICE_CHECK"}

EXPORTS = ["nr_status_string", "nr_params_default", "nr_index_load", "nr_index_free",
           "nr_index_info", "nr_set_params", "nr_encode", "nr_route", "nr_debug_clusters",
           "nr_search", "nr_search_logits", "nr_search_host", "nr_query_stats", "nr_last_stats",
           "nr_enable_timing", "nr_last_timing", "nr_kernel_launches", "nr_search_static",
           "nr_index_save", "nr_index_extract", "nr_index_thresholds", "nr_index_locate",
           "nr_centroid_dists", "nr_build_begin", "nr_build_encode", "nr_build_set_logits",
           "nr_build_finish", "nr_build_place", "nr_build_end", "nr_build_free",
           "nr_measure_gather", "nr_measure_read", "nr_bucket_scores", "nr_calib_observe", "nr_calib_fit_s_max",
           "nr_calib_fit_gate", "nr_calibrate"]


class NRError(RuntimeError):
    def __init__(self, call, status):
        super().__init__(f"{call} failed: {STATUS.get(status, status)}")
        self.status = status


class Params(ctypes.Structure):
    _fields_ = [("l_sel", ctypes.c_int), ("r_max", ctypes.c_int), ("s_max", ctypes.c_float),
                ("gate_m0", ctypes.c_float), ("gate_m1", ctypes.c_float),
                ("round_size", ctypes.c_int), ("t_low", ctypes.c_int), ("u_min", ctypes.c_int),
                ("f_min", ctypes.c_int), ("r_min", ctypes.c_int), ("alpha_front", ctypes.c_float),
                ("cent_mode", ctypes.c_int), ("n_bins", ctypes.c_int), ("b_batch", ctypes.c_int),
                ("b_min", ctypes.c_int), ("c_t_low", ctypes.c_int), ("c_u_min", ctypes.c_int),
                ("c_f_min", ctypes.c_int), ("c_alpha_front", ctypes.c_float),
                ("gate_n", ctypes.c_int), ("gate_x", ctypes.c_float * 16),
                ("gate_y", ctypes.c_float * 16), ("pipe_chunk", ctypes.c_int),
                ("refine_ctas", ctypes.c_int), ("nonempty_budget", ctypes.c_int),
                ("wait_limit_us", ctypes.c_int)]


class Stats(ctypes.Structure):
    _fields_ = [("nq", ctypes.c_int64), ("candidates", ctypes.c_int64), ("rounds", ctypes.c_int64),
                ("clusters", ctypes.c_int64), ("probes", ctypes.c_int64), ("scored", ctypes.c_int64)]


def lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(LIB_PATH)
        vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        L.nr_status_string.argtypes = [i32]
        L.nr_status_string.restype = ctypes.c_char_p
        L.nr_params_default.argtypes = [ctypes.POINTER(Params)]
        L.nr_index_load.argtypes = [ctypes.c_char_p, i32, ctypes.POINTER(vp)]
        L.nr_index_free.argtypes = [vp]
        L.nr_index_free.restype = None
        L.nr_index_info.argtypes = [vp, vp]
        L.nr_set_params.argtypes = [vp, ctypes.POINTER(Params)]
        L.nr_encode.argtypes = [vp, vp, i64, vp, vp]
        L.nr_route.argtypes = [vp, vp, i64, i32, vp, vp, vp]
        L.nr_debug_clusters.argtypes = [vp, vp, i64, i32, i32, vp, vp, vp]
        L.nr_search.argtypes = [vp, vp, i64, i32, i32, i32, vp, vp, vp]
        L.nr_search_logits.argtypes = [vp, vp, vp, i64, i32, i32, i32, vp, vp, vp]
        L.nr_search_host.argtypes = [vp, vp, i64, i32, i32, i32, vp, vp, vp]
        L.nr_search_static.argtypes = [vp, vp, i64, i32, i32, i32, vp, vp, vp]
        L.nr_query_stats.argtypes = [vp, vp, i64, vp]
        L.nr_last_stats.argtypes = [vp, ctypes.POINTER(Stats)]
        L.nr_measure_gather.argtypes = [i32, i64, i32, i64, i32, ctypes.POINTER(ctypes.c_double)]
        L.nr_measure_read.argtypes = [i32, i64, i32, ctypes.POINTER(ctypes.c_double)]
        dp, fp = ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_float)
        L.nr_bucket_scores.argtypes = [vp, vp, i32, vp, i64, i32, vp, vp]
        L.nr_calib_observe.argtypes = [vp, vp, vp, i64, i32, vp, vp, vp, vp]
        L.nr_calib_fit_s_max.argtypes = [vp, i64, i32, ctypes.c_double, fp, dp, dp]
        L.nr_calib_fit_gate.argtypes = [vp, vp, i64, i32, ctypes.c_double, ctypes.POINTER(i32), vp, vp]
        L.nr_calibrate.argtypes = [vp, vp, vp, i64, i32, i32, ctypes.c_double, ctypes.c_double,
                                   ctypes.POINTER(Params), vp, vp]
        L.nr_enable_timing.argtypes = [vp, i32]
        L.nr_last_timing.argtypes = [vp, vp]
        L.nr_kernel_launches.argtypes = [vp]
        L.nr_kernel_launches.restype = i64
        L.nr_index_save.argtypes = [vp, ctypes.c_char_p]
        L.nr_index_thresholds.argtypes = [vp, vp]
        L.nr_index_extract.argtypes = [vp, vp, i64, ctypes.c_char_p, vp]
        L.nr_index_locate.argtypes = [vp, vp, i64, vp, vp]
        L.nr_centroid_dists.argtypes = [vp, vp, i64, vp, i32, vp, vp]
        L.nr_build_begin.argtypes = [vp, i64, vp, vp, vp, vp, vp, i32, ctypes.POINTER(vp)]
        L.nr_build_encode.argtypes = [vp, vp, i64, i64, vp]
        L.nr_build_set_logits.argtypes = [vp, vp, i64, i64, vp]
        L.nr_build_finish.argtypes = [vp, vp]
        L.nr_build_place.argtypes = [vp, vp, i64, i64, vp]
        L.nr_build_end.argtypes = [vp, ctypes.POINTER(vp)]
        L.nr_build_free.argtypes = [vp]
        L.nr_build_free.restype = None
        for name in EXPORTS:
            if name not in ("nr_status_string", "nr_index_free", "nr_kernel_launches",
                            "nr_build_free"):
                getattr(L, name).restype = i32
        _LIB = L
    return _LIB


def _check(call, st):
    if st != NR_OK:
        raise NRError(call, st)


def params(**kw) -> Params:
    p = Params()
    lib().nr_params_default(ctypes.byref(p))
    for k, v in kw.items():
        if k == "gate_curve":  # (xs, ys): the calibrated piecewise-linear M, or None
            xs, ys = (v if v is not None else ((), ()))
            if len(xs) != len(ys) or len(xs) > 16:
                raise ValueError("gate_curve: up to 16 (x, y) points")
            p.gate_n = len(xs)
            for i in range(16):
                p.gate_x[i] = float(xs[i]) if i < len(xs) else 0.0
                p.gate_y[i] = float(ys[i]) if i < len(ys) else 0.0
            continue
        if not hasattr(p, k):
            raise KeyError(k)
        setattr(p, k, v)
    return p


def measure_read(device, nbytes=8 << 30, reps=5) -> float:
    """GB/s at which the GPU reads a long array sequentially (nr_measure_read)."""
    v = ctypes.c_double()
    _check("nr_measure_read", lib().nr_measure_read(int(device), int(nbytes), int(reps), ctypes.byref(v)))
    return v.value


def measure_gather(device, rows, row_bytes, n=20_000_000, reps=5) -> float:
    """GB/s at which the GPU reads rows at random (nr_measure_gather)."""
    v = ctypes.c_double()
    _check("nr_measure_gather", lib().nr_measure_gather(int(device), int(rows), int(row_bytes),
                                                        int(n), int(reps), ctypes.byref(v)))
    return v.value


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def _arg(t, name, dtype, shape, device):
    """Checks a tensor argument against what the C ABI reads or writes through
    its pointer (dtype, row-major contiguous shape, the index's GPU or the
    host for device None) and returns it; a mismatch raises before any call."""
    import torch

    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor, got {type(t).__name__}")
    if t.dtype != dtype:
        raise ValueError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if t.dim() != len(shape) or any(w is not None and v != w for v, w in zip(t.shape, shape)):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {shape}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous (row-major)")
    if device is None:
        if t.is_cuda:
            raise ValueError(f"{name}: expected a host tensor")
    elif not t.is_cuda or t.device.index != device:
        raise ValueError(f"{name}: expected a tensor on cuda:{device}, got {t.device}")
    return t


def _stream(stream):
    import torch

    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


class Index:
    """A loaded index on one GPU."""

    def __init__(self, path: str | None, device: int = 0, _handle=None):
        if _handle is None:
            h = ctypes.c_void_p()
            _check("nr_index_load", lib().nr_index_load(path.encode(), device, ctypes.byref(h)))
        else:
            h = _handle
        self.h = h
        self.device = device
        info = np.zeros(8, np.int64)
        lib().nr_index_info(h, info.ctypes.data)
        (self.N, self.D, self.H, self.b, self.n_clusters, self.dtype_code, self.k_max,
         self.t) = (int(v) for v in info)

    def close(self):
        if self.h:
            lib().nr_index_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def row_bytes(self):
        return self.D * (1 if self.dtype_code == 0 else 4)

    def thresholds(self) -> np.ndarray:
        """The per-bit thresholds tau [b] (nr_index_thresholds)."""
        tau = np.empty(self.b, np.float32)
        _check("nr_index_thresholds", lib().nr_index_thresholds(self.h, tau.ctypes.data))
        return tau

    def save(self, path: str):
        """Write the index file (nr_index_save)."""
        _check("nr_index_save", lib().nr_index_save(self.h, path.encode()))

    def extract(self, codes, path: str):
        """Write the sub-index of the buckets of `codes` (nr_index_extract);
        returns (rows, clusters)."""
        c = np.ascontiguousarray(np.asarray(codes).reshape(-1), np.uint32)
        info = np.zeros(2, np.int64)
        _check("nr_index_extract", lib().nr_index_extract(self.h, c.ctypes.data, c.size,
                                                          path.encode(), info.ctypes.data))
        return int(info[0]), int(info[1])

    def locate(self, ids, stream=None):
        """Where the rows `ids` (device int64) are stored (nr_index_locate):
        int32 [n x 4] = (cluster, bucket code, first cluster of the bucket,
        clusters in the bucket), (-1, -1, -1, 0) for an unknown id."""
        import torch

        ids = _arg(ids.reshape(-1).to(torch.int64).contiguous(), "ids", torch.int64, (None,),
                   self.device)
        out = torch.empty((ids.numel(), 4), dtype=torch.int32, device=self._dev())
        _check("nr_index_locate", lib().nr_index_locate(self.h, _ptr(ids), ids.numel(), _ptr(out),
                                                        _stream(stream)))
        return out

    def centroid_dists(self, logits, clusters, stream=None):
        """Distances of each query's logits to its listed clusters
        (nr_centroid_dists): fp32 [nq x m], +inf for -1 pads."""
        import torch

        clusters = _arg(clusters.to(torch.int32).contiguous(), "clusters", torch.int32,
                        (None, None), self.device)
        nq, m = clusters.shape
        self._logits(logits, nq)
        out = torch.empty((nq, m), dtype=torch.float32, device=self._dev())
        _check("nr_centroid_dists", lib().nr_centroid_dists(self.h, _ptr(logits), nq, _ptr(clusters), m,
                                                            _ptr(out), _stream(stream)))
        return out

    def set_params(self, p: Params | None = None, **kw):
        if p is None:
            p = params(**kw)
        _check("nr_set_params", lib().nr_set_params(self.h, ctypes.byref(p)))
        return p

    def _dev(self):
        import torch

        return torch.device("cuda", self.device)

    def _rows(self, x, name="queries", device=-1):
        """[n x D] rows of the index dtype on this index's GPU (device -1) or the host (None)."""
        import torch

        dt = torch.uint8 if self.dtype_code == 0 else torch.float32
        return _arg(x, name, dt, (None, self.D), self.device if device == -1 else device)

    def _logits(self, lg, nq=None):
        import torch

        return _arg(lg, "logits", torch.float32, (nq, self.b), self.device)

    def _outs(self, out, nq, k, device=-1):
        import torch

        dev = self.device if device == -1 else device
        ids, d = out
        return (_arg(ids, "out ids", torch.int64, (nq, k), dev),
                _arg(d, "out dists", torch.float32, (nq, k), dev))

    def encode(self, x, stream=None):
        import torch

        x = self._rows(x, "x")
        out = torch.empty((x.shape[0], self.b), dtype=torch.float32, device=self._dev())
        _check("nr_encode", lib().nr_encode(self.h, _ptr(x), x.shape[0], _ptr(out), _stream(stream)))
        return out

    def route(self, logits, P, stream=None):
        import torch

        logits = self._logits(logits)
        nq = logits.shape[0]
        codes = torch.empty((nq, P), dtype=torch.int32, device=self._dev())
        nprobe = torch.empty(nq, dtype=torch.int32, device=self._dev())
        _check("nr_route", lib().nr_route(self.h, _ptr(logits), nq, P, _ptr(codes), _ptr(nprobe),
                                          _stream(stream)))
        return codes, nprobe

    def debug_clusters(self, logits, P, C, stream=None):
        import torch

        logits = self._logits(logits)
        nq = logits.shape[0]
        cl = torch.empty((nq, P + C), dtype=torch.int32, device=self._dev())
        ncl = torch.empty(nq, dtype=torch.int32, device=self._dev())
        _check("nr_debug_clusters", lib().nr_debug_clusters(self.h, _ptr(logits), nq, P, C, _ptr(cl),
                                                            _ptr(ncl), _stream(stream)))
        return cl, ncl

    def _outputs(self, nq, k):
        import torch

        return (torch.empty((nq, k), dtype=torch.int64, device=self._dev()),
                torch.empty((nq, k), dtype=torch.float32, device=self._dev()))

    def search(self, queries, k, P, C, out=None, stream=None):
        nq = self._rows(queries).shape[0]
        ids, d = self._outs(out, nq, k) if out is not None else self._outputs(nq, k)
        _check("nr_search", lib().nr_search(self.h, _ptr(queries), nq, k, P, C, _ptr(ids), _ptr(d),
                                            _stream(stream)))
        return ids, d

    def search_logits(self, queries, logits, k, P, C, out=None, stream=None):
        nq = self._rows(queries).shape[0]
        self._logits(logits, nq)
        ids, d = self._outs(out, nq, k) if out is not None else self._outputs(nq, k)
        _check("nr_search_logits", lib().nr_search_logits(self.h, _ptr(queries), _ptr(logits), nq, k,
                                                          P, C, _ptr(ids), _ptr(d), _stream(stream)))
        return ids, d

    def search_host(self, queries, k, P, C, out=None, stream=None):
        """queries, and the outputs, are host tensors (pinned for full bandwidth)."""
        import torch

        nq = self._rows(queries, device=None).shape[0]
        if out is None:
            out = (torch.empty((nq, k), dtype=torch.int64), torch.empty((nq, k), dtype=torch.float32))
        ids, d = self._outs(out, nq, k, device=None)
        _check("nr_search_host", lib().nr_search_host(self.h, _ptr(queries), nq, k, P, C, _ptr(ids),
                                                      _ptr(d), _stream(stream)))
        return ids, d

    def search_static(self, queries, k, P, C, out=None, stream=None):
        """nr_search without any allocation inside the call: scratch comes from
        the library's fixed 32 MiB device array (see include/neuroute.h)."""
        nq = self._rows(queries).shape[0]
        ids, d = self._outs(out, nq, k) if out is not None else self._outputs(nq, k)
        _check("nr_search_static", lib().nr_search_static(self.h, _ptr(queries), nq, k, P, C,
                                                          _ptr(ids), _ptr(d), _stream(stream)))
        return ids, d

    def query_stats(self, nq, stream=None):
        import torch

        # per query: candidates, rounds, |L|, probes, centroid distances evaluated
        st = torch.empty((nq, 5), dtype=torch.int64, device=self._dev())
        _check("nr_query_stats", lib().nr_query_stats(self.h, _ptr(st), nq, _stream(stream)))
        return st

    def last_stats(self) -> Stats:
        s = Stats()
        _check("nr_last_stats", lib().nr_last_stats(self.h, ctypes.byref(s)))
        return s

    def enable_timing(self, on=True):
        _check("nr_enable_timing", lib().nr_enable_timing(self.h, 1 if on else 0))

    def last_timing(self):
        ms = np.zeros(4, np.float32)
        _check("nr_last_timing", lib().nr_last_timing(self.h, ms.ctypes.data))
        return {"encode": float(ms[0]), "route": float(ms[1]), "select": float(ms[2]),
                "refine": float(ms[3])}

    def kernel_launches(self) -> int:
        return int(lib().nr_kernel_launches(self.h))


class Builder:
    """A GPU index build (neuroute_build.h): pass 1 gives every row's logits
    (encode or set_logits), finish() builds thresholds, codes, clusters and
    the CSR levels, pass 2 places the rows, end() returns the Index.

    cfg is a ctypes structure with the fields of nr_build_config (the host
    builder's Config has the same layout); weights = (W1, b1, W2, b2[, middle
    layers ((W, b), ...)]) fp32."""

    def __init__(self, cfg, N: int, weights, device: int = 0):
        W1, b1, W2, b2 = (np.ascontiguousarray(w, np.float32) for w in weights[:4])
        mid = weights[4] if len(weights) > 4 else ()
        Wm = np.ascontiguousarray(np.concatenate(
            [np.concatenate([np.asarray(W, np.float32).ravel(), np.asarray(bb, np.float32).ravel()])
             for W, bb in mid]) if mid else np.zeros(1, np.float32))
        h = ctypes.c_void_p()
        _check("nr_build_begin", lib().nr_build_begin(
            ctypes.byref(cfg), N, W1.ctypes.data, b1.ctypes.data, W2.ctypes.data, b2.ctypes.data,
            Wm.ctypes.data if mid else None, device, ctypes.byref(h)))
        self.h, self.N, self.device, self.b = h, N, device, cfg.b

    def encode(self, rows, row0: int, stream=None):
        """Logits of rows [row0, row0 + len(rows)) from a CUDA tensor [n x D]."""
        _check("nr_build_encode", lib().nr_build_encode(self.h, _ptr(rows), row0, rows.shape[0],
                                                         _stream(stream)))

    def set_logits(self, logits, row0: int, stream=None):
        """Given logits [n x b] fp32 (CUDA tensor) of rows [row0, row0 + n)."""
        _check("nr_build_set_logits", lib().nr_build_set_logits(self.h, _ptr(logits), row0,
                                                                 logits.shape[0], _stream(stream)))

    def finish(self):
        info = np.zeros(5, np.int64)
        _check("nr_build_finish", lib().nr_build_finish(self.h, info.ctypes.data))
        return {"n_clusters": int(info[0]), "n_buckets": int(info[1]), "max_bucket": int(info[2]),
                "max_cluster": int(info[3]), "single_cluster_buckets": int(info[4])}

    def place(self, rows, row0: int, stream=None):
        """Store rows [row0, row0 + len(rows)) from a CUDA tensor [n x D]."""
        _check("nr_build_place", lib().nr_build_place(self.h, _ptr(rows), row0, rows.shape[0],
                                                      _stream(stream)))

    def end(self) -> Index:
        out = ctypes.c_void_p()
        h, self.h = self.h, None
        _check("nr_build_end", lib().nr_build_end(h, ctypes.byref(out)))
        return Index(None, self.device, _handle=out)

    def close(self):
        if self.h:
            lib().nr_build_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

"""ctypes binding of the NeuRoute query-path oracle (``oracle.cpp``).

Test infrastructure: only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use it. The product library never imports it.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None

c_i64p = ctypes.POINTER(ctypes.c_int64)


class Params(ctypes.Structure):
    _fields_ = [("l_sel", ctypes.c_int), ("r_max", ctypes.c_int), ("s_max", ctypes.c_float),
                ("gate_m0", ctypes.c_float), ("gate_m1", ctypes.c_float),
                ("round_size", ctypes.c_int), ("t_low", ctypes.c_int), ("u_min", ctypes.c_int),
                ("f_min", ctypes.c_int), ("r_min", ctypes.c_int), ("alpha_front", ctypes.c_float),
                ("cent_mode", ctypes.c_int), ("n_bins", ctypes.c_int), ("b_batch", ctypes.c_int),
                ("b_min", ctypes.c_int), ("c_t_low", ctypes.c_int), ("c_u_min", ctypes.c_int),
                ("c_f_min", ctypes.c_int), ("c_alpha_front", ctypes.c_float),
                ("gate_n", ctypes.c_int), ("gate_x", ctypes.c_float * 16),
                ("gate_y", ctypes.c_float * 16), ("nonempty_budget", ctypes.c_int)]


def lib():
    global _LIB
    if _LIB is None:
        path = os.path.join(_HERE, "liboracle.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(path)
        vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        L.or_params_default.argtypes = [ctypes.POINTER(Params)]
        L.or_index_load.argtypes = [ctypes.c_char_p, ctypes.c_char_p, i32]
        L.or_index_load.restype = vp
        L.or_index_free.argtypes = [vp]
        L.or_index_info.argtypes = [vp, vp]
        for name in ("or_index_bkt_off", "or_index_cl_off", "or_index_ids", "or_index_tau",
                     "or_index_cent"):
            getattr(L, name).argtypes = [vp]
            getattr(L, name).restype = vp
        L.or_encode.argtypes = [vp, vp, i64, vp, i32]
        L.or_encode_weights.argtypes = [i32, i32, i32, i32, ctypes.c_float, vp, vp, vp, vp, vp, i64,
                                        vp, i32]
        L.or_encode_weights.restype = None
        L.or_encode_mlp.argtypes = [i32, i32, i32, i32, i32, vp, ctypes.c_float, vp, vp, vp, vp, vp,
                                    vp, i64, vp, i32]
        L.or_encode_mlp.restype = None
        L.or_index_mid.argtypes = [vp, vp]
        L.or_index_mid.restype = i32
        L.or_probe_order.argtypes = [i32, vp, i32, ctypes.POINTER(Params), vp]
        L.or_probe_order.restype = i32
        L.or_probe_order_allsubsets.argtypes = [i32, vp, i32, ctypes.POINTER(Params), vp]
        L.or_probe_order_allsubsets.restype = i32
        L.or_probe_list.argtypes = [i32, vp, vp, i32, ctypes.POINTER(Params), vp, vp, vp]
        L.or_probe_list.restype = i32
        L.or_cluster_list.argtypes = [vp, vp, vp, i32, i32, ctypes.POINTER(Params), vp, vp, vp,
                                      vp]
        L.or_cluster_list_seq.argtypes = [vp, vp, vp, vp, i32, i32, ctypes.POINTER(Params), vp, vp,
                                          vp, vp, vp]
        L.or_cluster_list_seq.restype = i32
        L.or_cluster_list.restype = i32
        L.or_refine_stream.argtypes = [i32, i32, vp, vp, vp, i64, i32, ctypes.POINTER(Params),
                                       vp, vp, vp]
        L.or_search.argtypes = [vp, vp, vp, i64, i32, i32, i32, ctypes.POINTER(Params), vp, vp,
                                vp, i32]
        L.or_search.restype = i32
        L.or_bruteforce.argtypes = [i32, i32, vp, i64, vp, i64, i32, vp, vp, i32]
        L.or_probe_list_index.argtypes = [vp, vp, i32, ctypes.POINTER(Params), vp, vp]
        L.or_probe_list_index.restype = i32
        L.or_centroid_dist.argtypes = [vp, vp, i64]
        L.or_centroid_dist.restype = ctypes.c_float
        L.or_gate_margin.argtypes = [ctypes.POINTER(Params), ctypes.c_float]
        L.or_gate_margin.restype = ctypes.c_float
        _LIB = L
    return _LIB


def _p(a):
    return None if a is None else a.ctypes.data


def params(**kw) -> Params:
    p = Params()
    lib().or_params_default(ctypes.byref(p))
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


def nthreads_default() -> int:
    return os.cpu_count() or 1


class Index:
    """An index file loaded by the oracle's own reader."""

    def __init__(self, path: str):
        err = ctypes.create_string_buffer(256)
        h = lib().or_index_load(path.encode(), err, 256)
        if not h:
            raise RuntimeError(f"oracle: cannot load {path}: {err.value.decode()}")
        self.h = h
        info = np.zeros(8, np.int64)
        lib().or_index_info(h, info.ctypes.data)
        (self.N, self.D, self.H, self.b, self.n_clusters, self.dtype_code, self.k_max,
         self.t) = (int(v) for v in info)
        w = np.zeros(8, np.int32)
        self.mid = tuple(int(v) for v in w[: lib().or_index_mid(h, w.ctypes.data)])

    def close(self):
        if self.h:
            lib().or_index_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _arr(self, fn, n, dt):
        ptr = getattr(lib(), fn)(self.h)
        buf = (ctypes.c_char * (n * np.dtype(dt).itemsize)).from_address(ptr)
        return np.frombuffer(buf, dtype=dt).copy()

    def bkt_off(self):
        return self._arr("or_index_bkt_off", (1 << self.b) + 1, np.uint32)

    def cl_off(self):
        return self._arr("or_index_cl_off", self.n_clusters + 1, np.uint32)

    def ids(self):
        return self._arr("or_index_ids", self.N, np.uint32)

    def tau(self):
        return self._arr("or_index_tau", self.b, np.float32)

    def centroids(self):
        return self._arr("or_index_cent", self.n_clusters * self.b, np.float32).reshape(-1, self.b)

    def encode(self, x: np.ndarray, nthreads=None) -> np.ndarray:
        x = np.ascontiguousarray(x)
        out = np.empty((x.shape[0], self.b), np.float32)
        lib().or_encode(self.h, x.ctypes.data, x.shape[0], out.ctypes.data,
                        nthreads or nthreads_default())
        return out

    def cluster_list(self, logit, codes, C, p: Params):
        logit = np.ascontiguousarray(logit, np.float32)
        codes = np.ascontiguousarray(codes, np.uint32)
        L = np.empty(len(codes) + C, np.int32)
        dL = np.empty(len(codes) + C, np.float32)
        ndir = np.zeros(1, np.int32)
        n = lib().or_cluster_list(self.h, logit.ctypes.data, codes.ctypes.data, len(codes), C,
                                  ctypes.byref(p), L.ctypes.data, dL.ctypes.data, ndir.ctypes.data,
                                  None)
        if n < 0:
            raise RuntimeError("oracle: out-of-range index in file")
        return L[:n].copy(), dL[:n].copy(), int(ndir[0])

    def cluster_list_seq(self, logit, codes, scores, C, p: Params, with_scored=False):
        """The sequential centroid stage (Algorithm 2): returns (L, dL, n_dir,
        n_batches), and the number of centroid distances evaluated after them
        when with_scored."""
        logit = np.ascontiguousarray(logit, np.float32)
        codes = np.ascontiguousarray(codes, np.uint32)
        scores = np.ascontiguousarray(scores, np.float32)
        L = np.empty(len(codes) + C, np.int32)
        dL = np.empty(len(codes) + C, np.float32)
        ndir = np.zeros(1, np.int32)
        nbat = np.zeros(1, np.int32)
        nsc = np.zeros(1, np.int64)
        n = lib().or_cluster_list_seq(self.h, logit.ctypes.data, codes.ctypes.data,
                                      scores.ctypes.data, len(codes), C, ctypes.byref(p),
                                      L.ctypes.data, dL.ctypes.data, ndir.ctypes.data,
                                      nbat.ctypes.data, nsc.ctypes.data)
        if n < 0:
            raise RuntimeError("oracle: out-of-range index in file")
        out = (L[:n].copy(), dL[:n].copy(), int(ndir[0]), int(nbat[0]))
        return out + (int(nsc[0]),) if with_scored else out

    def probe_list(self, logit, P, p: Params):
        """(codes, keys) of one query's probe list against this index (the
        non-empty budget skips empty buckets)."""
        logit = np.ascontiguousarray(logit, np.float32)
        codes = np.empty(max(P, 1), np.uint32)
        keys = np.empty(max(P, 1), np.uint64)
        n = lib().or_probe_list_index(self.h, logit.ctypes.data, P, ctypes.byref(p), codes.ctypes.data,
                                      keys.ctypes.data)
        return codes[:n].copy(), keys[:n].copy()

    def centroid_dist(self, logit, c: int) -> np.float32:
        """Distance of cluster c's centroid from the logits (the centroid
        stage's fmaf chain); +inf for c out of range."""
        logit = np.ascontiguousarray(logit, np.float32)
        return np.float32(lib().or_centroid_dist(self.h, logit.ctypes.data, int(c)))

    def search(self, queries, k, P, C, p: Params, logits=None, nthreads=None):
        queries = np.ascontiguousarray(queries)
        nq = queries.shape[0]
        ids = np.empty((nq, k), np.int64)
        d = np.empty((nq, k), np.float32)
        st = np.empty((nq, 5), np.int64)  # candidates, rounds, |L|, probes, distances evaluated
        lg = None if logits is None else np.ascontiguousarray(logits, np.float32)
        rc = lib().or_search(self.h, queries.ctypes.data, _p(lg), nq, k, P, C, ctypes.byref(p),
                             ids.ctypes.data, d.ctypes.data, st.ctypes.data,
                             nthreads or nthreads_default())
        if rc != 0:
            raise RuntimeError("oracle: out-of-range index in file")
        return ids, d, st


def mid_layers(weights):
    """The hidden layers after the first of an encoder given as (W1, b1, W2,
    b2) or (W1, b1, W2, b2, ((W, b), ...)): (widths, the concatenated W then b
    of each layer as the file stores them)."""
    mid = weights[4] if len(weights) > 4 else ()
    widths = [int(np.asarray(W).shape[0]) for W, _ in mid]
    flat = [np.concatenate([np.asarray(W, np.float32).ravel(), np.asarray(bb, np.float32).ravel()])
            for W, bb in mid]
    return widths, (np.concatenate(flat) if flat else np.zeros(0, np.float32))


def encode_weights(weights, in_scale: float, x: np.ndarray, nthreads=None) -> np.ndarray:
    """Logits of rows x under the encoder (W1, b1, W2, b2[, middle layers]),
    without an index."""
    W1, b1, W2, b2 = (np.ascontiguousarray(w, np.float32) for w in weights[:4])
    widths, Wm = mid_layers(weights)
    x = np.ascontiguousarray(x)
    H, D = W1.shape
    b = W2.shape[0]
    out = np.empty((x.shape[0], b), np.float32)
    w = (ctypes.c_int * max(1, len(widths)))(*widths)
    lib().or_encode_mlp(0 if x.dtype == np.uint8 else 1, D, H, b, len(widths), w, in_scale,
                        W1.ctypes.data, b1.ctypes.data, W2.ctypes.data, b2.ctypes.data,
                        Wm.ctypes.data, x.ctypes.data, x.shape[0], out.ctypes.data,
                        nthreads or nthreads_default())
    return out


def gate_margin(p: Params, x) -> np.float32:
    """M(x) under the parameters p."""
    return np.float32(lib().or_gate_margin(ctypes.byref(p), float(np.float32(x))))


def probe_order(sd, P, p: Params):
    sd = np.ascontiguousarray(sd, np.float32)
    keys = np.empty(max(P, 1), np.uint64)
    n = lib().or_probe_order(len(sd), sd.ctypes.data, P, ctypes.byref(p), keys.ctypes.data)
    return keys[:n].copy()


def probe_order_allsubsets(sd, P, p: Params):
    sd = np.ascontiguousarray(sd, np.float32)
    keys = np.empty(max(P, 1), np.uint64)
    n = lib().or_probe_order_allsubsets(len(sd), sd.ctypes.data, P, ctypes.byref(p),
                                        keys.ctypes.data)
    return keys[:n].copy()


def probe_list(logit, tau, P, p: Params):
    logit = np.ascontiguousarray(logit, np.float32)
    tau = np.ascontiguousarray(tau, np.float32)
    b = len(logit)
    codes = np.empty(max(P, 1), np.uint32)
    keys = np.empty(max(P, 1), np.uint64)
    perm = np.empty(b, np.int32)
    n = lib().or_probe_list(b, logit.ctypes.data, tau.ctypes.data, P, ctypes.byref(p),
                            codes.ctypes.data, keys.ctypes.data, perm.ctypes.data)
    return codes[:n].copy(), keys[:n].copy(), perm


def refine_stream(q, rows, ids, k, p: Params):
    q = np.ascontiguousarray(q)
    rows = np.ascontiguousarray(rows)
    ids = np.ascontiguousarray(ids, np.uint32)
    dtype = 0 if rows.dtype == np.uint8 else 1
    out_ids = np.empty(k, np.int64)
    out_d = np.empty(k, np.float32)
    st = np.zeros(2, np.int64)
    lib().or_refine_stream(dtype, rows.shape[1], q.ctypes.data, rows.ctypes.data, ids.ctypes.data,
                           rows.shape[0], k, ctypes.byref(p), out_ids.ctypes.data,
                           out_d.ctypes.data, st.ctypes.data)
    return out_ids, out_d, st


def bruteforce(base, queries, k, nthreads=None):
    base = np.ascontiguousarray(base)
    queries = np.ascontiguousarray(queries)
    dtype = 0 if base.dtype == np.uint8 else 1
    nq = queries.shape[0]
    ids = np.empty((nq, k), np.int64)
    d = np.empty((nq, k), np.float32)
    lib().or_bruteforce(dtype, base.shape[1], base.ctypes.data, base.shape[0], queries.ctypes.data,
                        nq, k, ids.ctypes.data, d.ctypes.data, nthreads or nthreads_default())
    return ids, d


def unpack_key(key):
    key = int(key)
    cost = np.array([key >> 32], np.uint32).view(np.float32)[0]
    return float(cost), (key >> 24) & 0xFF, key & 0xFFFFFF

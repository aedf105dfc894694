"""Calibration of the bucket-score cutoff S_max and the centroid gate margin
M(x) from held-out calibration queries (Sec. 3.4).

The targets are each calibration query's top-k from a high-recall run of the
same search (enlarged budgets, gate and early stop off), or any top-k list
the caller passes (exact k-NN, say). From where the targets are stored:

  score  the bucket enumeration's cost of the bucket holding a target: bit
         deviations delta_j = |l_j - tau_j| ranked by (delta_j, j), summed in
         fp32 over the ranks whose bit differs from the base code, in
         ascending rank (Algorithm 1);
  x      per query, the smallest centroid distance over every cluster of the
         target buckets that hold two or more clusters (single-cluster buckets
         bypass the gate, Sec. 3.4.2), undefined without one;
  y      the largest centroid distance of a gated target's own cluster, minus
         x: the margin that lets the farthest target through theta = x + M(x).

S_max is the score at sorted position ceil(coverage * m) - 1 of the m target
scores. M is fitted on equal-frequency bins of the queries sorted by (x, y):
bin i holds positions [floor(i n / B), floor((i + 1) n / B)) with B =
min(n_bins, n); its point is (x at the bin's lower-median position, the
bin's y at sorted position ceil(q m) - 1); points with equal x merge (largest
y); the curve is the running maximum of the y's, the smallest non-decreasing
curve on or above every bin's quantile. A single point (x0, y0) gives the
flat curve through (x0, y0) and (next float above x0, y0).

Every step runs in the library (nr_calib_observe, nr_calib_fit_s_max,
nr_calib_fit_gate: the observations on the GPU, the fits on the host); this
module only marshals arguments.
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import neuroute as nr


def bucket_scores(logits, tau, codes, stream=None) -> np.ndarray:
    """Cost of bucket codes[q, t] for query q (fp32 [nq x k]); nan where the
    code is negative (nr_bucket_scores on the GPU)."""
    import torch

    dev = torch.device("cuda", torch.cuda.current_device())
    lg = torch.as_tensor(np.asarray(logits, np.float32), device=dev).contiguous()
    tu = torch.as_tensor(np.asarray(tau, np.float32), device=dev).contiguous()
    cd = torch.as_tensor(np.asarray(codes, np.int64).astype(np.int32), device=dev).contiguous()
    nq, b = lg.shape
    k = cd.shape[1]
    out = torch.empty((nq, k), dtype=torch.float32, device=dev)
    st = nr.lib().nr_bucket_scores(nr._ptr(lg), nr._ptr(tu), b, nr._ptr(cd), nq, k, nr._ptr(out),
                                   nr._stream(stream))
    nr._check("nr_bucket_scores", st)
    return out.cpu().numpy()


def observations(ix: "nr.Index", logits, targets, stream=None):
    """(scores [nq x k], x [nq], y [nq]) as numpy fp32 for device logits
    [nq x b] and device int64 targets [nq x k] (-1 = none)."""
    import torch

    nq, k = targets.shape
    dev = logits.device
    lg = nr._arg(logits, "logits", torch.float32, (nq, ix.b), ix.device)
    tg = nr._arg(targets, "targets", torch.int64, (nq, k), ix.device)
    sc = torch.empty((nq, k), dtype=torch.float32, device=dev)
    x = torch.empty(nq, dtype=torch.float32, device=dev)
    y = torch.empty(nq, dtype=torch.float32, device=dev)
    st = nr.lib().nr_calib_observe(ix.h, nr._ptr(lg), nr._ptr(tg), nq, k, nr._ptr(sc), nr._ptr(x),
                                   nr._ptr(y), nr._stream(stream))
    nr._check("nr_calib_observe", st)
    return sc.cpu().numpy(), x.cpu().numpy(), y.cpu().numpy()


def fit_s_max(scores, coverage: float):
    """(S_max, fraction of target pairs covered, fraction of queries whose
    every target is covered); (None, 0, 0) without scores."""
    scores = np.ascontiguousarray(np.asarray(scores, np.float32))
    if scores.size == 0:
        return None, 0.0, 0.0
    scores = scores.reshape(len(scores), -1)
    t = ctypes.c_float()
    pc, qc = ctypes.c_double(), ctypes.c_double()
    st = nr.lib().nr_calib_fit_s_max(scores.ctypes.data, scores.shape[0], max(1, scores.shape[1]),
                                     float(coverage), ctypes.byref(t), ctypes.byref(pc),
                                     ctypes.byref(qc))
    nr._check("nr_calib_fit_s_max", st)
    if np.isnan(t.value):
        return None, 0.0, 0.0
    return np.float32(t.value), pc.value, qc.value


def fit_gate(x, y, n_bins: int = 16, q: float = 0.95):
    """The calibrated margin curve (xs, ys), up to 16 points, or None without
    observations."""
    if not 1 <= n_bins <= 16:
        raise ValueError("n_bins: 1..16")
    x = np.ascontiguousarray(x, np.float32)
    y = np.ascontiguousarray(y, np.float32)
    n = ctypes.c_int()
    gx, gy = np.zeros(16, np.float32), np.zeros(16, np.float32)
    st = nr.lib().nr_calib_fit_gate(x.ctypes.data, y.ctypes.data, x.size, int(n_bins), float(q),
                                    ctypes.byref(n), gx.ctypes.data, gy.ctypes.data)
    nr._check("nr_calib_fit_gate", st)
    if n.value == 0:
        return None
    return tuple(float(v) for v in gx[:n.value]), tuple(float(v) for v in gy[:n.value])


def targets_high_recall(ix: "nr.Index", queries, logits, k: int, P: int, C: int, stream=None):
    """Top-k of the search itself under budgets (P, C) with the gate and the
    early stop off; the index's parameters are reset to the defaults after."""
    ix.set_params(t_low=0)
    try:
        ids, _ = ix.search_logits(queries, logits, k, P, C, stream=stream)
    finally:
        ix.set_params()
    return ids


def calibrate(ix: "nr.Index", queries, k: int = 10, P: int = 1024, C: int = 4096, targets=None,
              n_bins: int = 16, quantile: float = 0.95, coverage: float = 0.99, stream=None):
    """Calibrate M(x) and S_max on device calibration queries [nq x D].
    Returns a dict: gate_curve (xs, ys) or None, s_max, pair and query
    coverage at s_max, the number of queries with an x, and the raw
    observations (scores, x, y)."""
    logits = ix.encode(queries, stream)
    if targets is None:
        targets = targets_high_recall(ix, queries, logits, k, P, C, stream)
    scores, x, y = observations(ix, logits, targets, stream)
    s_max, pair_cov, query_cov = fit_s_max(scores, coverage)
    return {"gate_curve": fit_gate(x, y, n_bins, quantile), "s_max": s_max, "pair_coverage": pair_cov,
            "query_coverage": query_cov, "n_gated": int((~np.isnan(x)).sum()), "scores": scores,
            "x": x, "y": y}

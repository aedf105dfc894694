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

Locations and centroid distances come from the library (nr_index_locate,
nr_centroid_dists); the scores and the fits are host arithmetic on at most a
few hundred thousand numbers, done once per index.
"""
from __future__ import annotations

import math

import numpy as np

from . import neuroute as nr


def bucket_scores(logits: np.ndarray, tau: np.ndarray, codes: np.ndarray) -> np.ndarray:
    """Cost of bucket codes[q, t] for query q (fp32 [nq x k]); nan where the
    code is negative."""
    logits = np.asarray(logits, np.float32)
    tau = np.asarray(tau, np.float32)
    codes = np.asarray(codes, np.int64)
    nq, b = logits.shape
    delta = np.abs(logits - tau[None, :])
    u0 = ((logits >= tau[None, :]).astype(np.int64) << np.arange(b, dtype=np.int64)).sum(axis=1)
    ranks = np.argsort(delta, axis=1, kind="stable")          # ties: lower bit first
    diff = codes ^ u0[:, None]
    rows = np.arange(nq)
    s = np.zeros(codes.shape, np.float32)
    for r in range(b):
        j = ranks[:, r]
        flip = ((diff >> j[:, None]) & 1).astype(bool)
        s = np.where(flip, s + delta[rows, j][:, None], s)
    return np.where(codes >= 0, s, np.float32(np.nan)).astype(np.float32)


def observations(ix: "nr.Index", logits, targets, stream=None):
    """(scores [nq x k], x [nq], y [nq]) as numpy fp32 for device logits
    [nq x b] and device int64 targets [nq x k] (-1 = none)."""
    import torch

    nq, k = targets.shape
    loc = ix.locate(targets, stream).view(nq, k, 4)
    loc_h = loc.cpu().numpy()
    lg = logits.cpu().numpy()
    found = loc_h[..., 0] >= 0
    scores = bucket_scores(lg, ix.thresholds(), np.where(found, loc_h[..., 1], -1))
    gated = found & (loc_h[..., 3] >= 2)
    j = np.arange(ix.k_max, dtype=np.int32)
    members = np.where(gated[..., None] & (j < loc_h[..., 3:4]), loc_h[..., 2:3] + j, -1)
    dev = logits.device
    d_all = ix.centroid_dists(logits, torch.from_numpy(members.reshape(nq, -1)).to(dev), stream)
    d_own = ix.centroid_dists(logits, torch.from_numpy(np.where(gated, loc_h[..., 0], -1)).to(dev),
                              stream)
    d_all, d_own = d_all.cpu().numpy(), d_own.cpu().numpy()
    has = gated.any(axis=1)
    x = d_all.min(axis=1)
    far = np.where(gated, d_own, np.float32(-np.inf)).max(axis=1)
    with np.errstate(invalid="ignore"):  # queries without a gated target: -inf - inf
        y = (far - x).astype(np.float32)
    nan = np.float32(np.nan)
    return scores, np.where(has, x, nan).astype(np.float32), np.where(has, y, nan).astype(np.float32)


def fit_s_max(scores, coverage: float):
    """(S_max, fraction of target pairs covered, fraction of queries whose
    every target is covered); (None, 0, 0) without scores."""
    scores = np.asarray(scores, np.float32)
    valid = ~np.isnan(scores)
    flat = np.sort(scores[valid])
    m = flat.size
    if m == 0:
        return None, 0.0, 0.0
    t = flat[min(m - 1, max(0, math.ceil(coverage * m) - 1))]
    pairs = int((flat <= t).sum()) / m
    has = valid.any(axis=1)
    worst = np.where(valid, scores, np.float32(-np.inf)).max(axis=1)
    return np.float32(t), pairs, int((worst[has] <= t).sum()) / int(has.sum())


def fit_gate(x, y, n_bins: int = 16, q: float = 0.95):
    """The calibrated margin curve (xs, ys), up to 16 points, or None without
    observations."""
    if not 1 <= n_bins <= 16:
        raise ValueError("n_bins: 1..16")
    x, y = np.asarray(x, np.float32), np.asarray(y, np.float32)
    keep = ~np.isnan(x)
    x, y = x[keep], y[keep]
    n = x.size
    if n == 0:
        return None
    order = np.lexsort((y, x))
    x, y = x[order], y[order]
    B = min(n_bins, n)
    px, py = [], []
    for i in range(B):
        lo, hi = i * n // B, (i + 1) * n // B
        m = hi - lo
        xm = x[lo + (m - 1) // 2]
        yq = np.sort(y[lo:hi])[min(m - 1, max(0, math.ceil(q * m) - 1))]
        if px and px[-1] == xm:
            py[-1] = max(py[-1], yq)
        else:
            px.append(xm)
            py.append(yq)
    ys = np.maximum.accumulate(np.array(py, np.float32))
    xs = np.array(px, np.float32)
    if xs.size == 1:
        xs = np.array([xs[0], np.nextafter(xs[0], np.float32(np.inf))], np.float32)
        ys = np.array([ys[0], ys[0]], np.float32)
    return tuple(float(v) for v in xs), tuple(float(v) for v in ys)


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

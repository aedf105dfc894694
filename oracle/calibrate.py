"""Calibration of the bucket-score cutoff S_max and the centroid gate margin
M(x) (Sec. 3.4), written step by step as plain Python loops.

TEST INFRASTRUCTURE: only the tests use it. It shares nothing with the
package's calibration; both take the same definitions:

  targets    a top-k list per calibration query (row ids, -1 = none), from a
             high-recall run of the search or from exact k-NN.
  score      of a target: the summed deviation of the flip set that turns the
             query's base code u0 into the code of the target's bucket, the
             bucket enumeration's cost (Algorithm 1): ranks by (delta_j, j),
             F = ranks whose bit differs, fp32 sum over F in ascending rank.
  x          per query: the smallest centroid distance over every cluster of
             every target bucket that holds two or more clusters (buckets of
             one cluster bypass the gate, Sec. 3.4.2); undefined when there is
             none.
  y          per query: the largest centroid distance of a target's own
             cluster among those buckets, minus x (one fp32 subtraction): the
             margin the farthest target needs to pass theta = x + M(x).
  S_max      the smallest score t with at least a fraction `coverage` of all
             (query, target) pairs at score <= t: the pair scores sorted, the
             entry at position ceil(coverage * m) - 1.
  M(x)       equal-frequency bins of the queries sorted by (x, y): bin i holds
             sorted positions [floor(i n / B), floor((i + 1) n / B)), B =
             min(n_bins, n). Its point is (x at the bin's lower-median position,
             the q-quantile of the bin's y = sorted entry ceil(q m) - 1).
             Points with equal x merge (largest y). The curve is the running
             maximum of the y's (the smallest non-decreasing curve on or above
             every bin's quantile); a single point (x0, y0) becomes the flat
             curve through (x0, y0) and (next float above x0, y0).
"""
from __future__ import annotations

import bisect
import math

import numpy as np


def bucket_score(logit, tau, code: int) -> np.float32:
    """The bucket enumeration's cost of the bucket `code` for one query."""
    b = len(tau)
    delta = [np.float32(abs(np.float32(logit[j]) - np.float32(tau[j]))) for j in range(b)]
    u0 = 0
    for j in range(b):
        if np.float32(logit[j]) >= np.float32(tau[j]):
            u0 |= 1 << j
    ranks = sorted(range(b), key=lambda j: (delta[j], j))
    diff = int(code) ^ u0
    s = np.float32(0.0)
    for r in range(b):
        if (diff >> ranks[r]) & 1:
            s = np.float32(s + delta[ranks[r]])
    return s


def locate(ix, ids):
    """Per id: (cluster, bucket code, first cluster of the bucket, clusters
    in the bucket), or (-1, -1, -1, 0) when the id is not stored."""
    stored = ix.ids()
    pos = {int(v): p for p, v in enumerate(stored)}
    cl_off = [int(v) for v in ix.cl_off()]
    bkt_off = [int(v) for v in ix.bkt_off()]
    out = []
    for i in ids:
        p = pos.get(int(i), -1) if int(i) >= 0 else -1
        if p < 0:
            out.append((-1, -1, -1, 0))
            continue
        c = bisect.bisect_right(cl_off, p) - 1
        u = bisect.bisect_right(bkt_off, c) - 1  # the last bucket starting at or before c
        out.append((c, u, bkt_off[u], bkt_off[u + 1] - bkt_off[u]))
    return out


def observations(ix, logits, targets):
    """Per query: the scores of its targets (nan where none), x and y (nan
    where undefined)."""
    tau = ix.tau()
    nq, k = targets.shape
    scores = np.full((nq, k), np.nan, np.float32)
    x = np.full(nq, np.nan, np.float32)
    y = np.full(nq, np.nan, np.float32)
    for q in range(nq):
        loc = locate(ix, targets[q])
        for t in range(k):
            if loc[t][0] >= 0:
                scores[q, t] = bucket_score(logits[q], tau, loc[t][1])
        best = None
        far = None
        for t in range(k):
            c, _, first, count = loc[t]
            if c < 0 or count < 2:
                continue
            for cc in range(first, first + count):
                d = ix.centroid_dist(logits[q], cc)
                if best is None or d < best:
                    best = d
            d = ix.centroid_dist(logits[q], c)
            if far is None or d > far:
                far = d
        if best is not None:
            x[q] = best
            y[q] = np.float32(far - best)
    return scores, x, y


def fit_s_max(scores, coverage: float):
    """(S_max, fraction of pairs covered, fraction of queries with every
    target covered)."""
    flat = sorted(float(s) for s in np.asarray(scores).reshape(-1) if not math.isnan(s))
    m = len(flat)
    if m == 0:
        return None, 0.0, 0.0
    pos = min(m - 1, max(0, math.ceil(coverage * m) - 1))
    t = flat[pos]
    pairs = sum(1 for s in flat if s <= t) / m
    nq_with, covered = 0, 0
    for row in np.asarray(scores):
        vals = [float(s) for s in row if not math.isnan(s)]
        if vals:
            nq_with += 1
            covered += all(s <= t for s in vals)
    return np.float32(t), pairs, covered / nq_with


def fit_gate(x, y, n_bins: int, q: float):
    """The calibrated margin curve as (xs, ys), or None without observations."""
    obs = sorted((float(a), float(c)) for a, c in zip(x, y) if not math.isnan(a))
    n = len(obs)
    if n == 0:
        return None
    B = min(n_bins, n)
    pts = []
    for i in range(B):
        lo, hi = i * n // B, (i + 1) * n // B
        m = hi - lo
        xm = obs[lo + (m - 1) // 2][0]
        ys = sorted(c for _, c in obs[lo:hi])
        yq = ys[min(m - 1, max(0, math.ceil(q * m) - 1))]
        if pts and pts[-1][0] == xm:
            pts[-1] = (xm, max(pts[-1][1], yq))
        else:
            pts.append((xm, yq))
    xs, ys = [], []
    run = -math.inf
    for a, c in pts:
        run = max(run, c)
        xs.append(np.float32(a))
        ys.append(np.float32(run))
    if len(xs) == 1:
        xs.append(np.nextafter(xs[0], np.float32(np.inf)))
        ys.append(ys[0])
    return tuple(xs), tuple(ys)

"""The selective similarity-preservation loss of NeuRoute's encoder training,
written out plainly in float64 numpy (test infrastructure: only the tests
use it; the package's training code shares nothing with it).

Definitions (paper Sec. 3.2.2 and Sec. 4.5.1):
  * pairwise Euclidean distances of a mini-batch: S_emb(i, j) = ||x_i - x_j||_2
    of the embeddings, S_lat(i, j) = ||l_i - l_j||_2 of their latents;
  * rho = sqrt(L_dim / E_dim), gamma the scaling coefficient (0.6);
  * Mask(i, j) = 1 iff i != j and (S_emb(i, j) <= tau_emb or
    S_lat(i, j) <= gamma rho tau_emb) (Eq. "equation8");
  * L_sim = sum_ij Mask(i, j) (S_lat(i, j) - gamma rho S_emb(i, j))^2 /
    sum(Mask) (Eq. "similarityconfig");
  * tau_emb is chosen per mini-batch so that only the closest 0.5% of the
    pairs satisfy S_emb <= tau_emb (Sec. 4.5.1). Reading taken here: over the
    B (B - 1) / 2 unordered pairs i < j, tau_emb is the order statistic at
    sorted position ceil(q B (B - 1) / 2) - 1 with q = 0.005 (at least one
    pair), so that exactly that many pairs (more only on ties) fall within it.
"""
from __future__ import annotations

import math

import numpy as np


def pairwise_l2(X: np.ndarray) -> np.ndarray:
    """S(i, j) = ||x_i - x_j||_2 by explicit differences (float64)."""
    X = np.asarray(X, np.float64)
    diff = X[:, None, :] - X[None, :, :]
    return np.sqrt((diff * diff).sum(-1))


def tau_emb(S_emb: np.ndarray, q: float = 0.005) -> float:
    """The distance at which the closest fraction q of the unordered pairs
    (i < j) lie: the order statistic at position ceil(q n_pairs) - 1."""
    B = S_emb.shape[0]
    iu = np.triu_indices(B, 1)
    d = np.sort(S_emb[iu])
    k = max(1, math.ceil(q * d.size)) - 1
    return float(d[k])


def mask(S_emb: np.ndarray, S_lat: np.ndarray, tau: float, gamma: float, rho: float) -> np.ndarray:
    """Eq. "equation8": off-diagonal pairs close in either space."""
    B = S_emb.shape[0]
    m = (S_emb <= tau) | (S_lat <= gamma * rho * tau)
    m[np.arange(B), np.arange(B)] = False
    return m


def l_sim(S_emb: np.ndarray, S_lat: np.ndarray, M: np.ndarray, gamma: float, rho: float) -> float:
    """Eq. "similarityconfig": the masked mean squared discrepancy."""
    r = S_lat - gamma * rho * S_emb
    return float((M * r * r).sum() / M.sum())


def batch_loss(X: np.ndarray, L: np.ndarray, gamma: float = 0.6, q: float = 0.005):
    """L_sim of one mini-batch of embeddings X [B x E_dim] and latents
    L [B x L_dim]; returns (loss, tau_emb, mask)."""
    rho = math.sqrt(L.shape[1] / X.shape[1])
    Se, Sl = pairwise_l2(X), pairwise_l2(L)
    t = tau_emb(Se, q)
    M = mask(Se, Sl, t, gamma, rho)
    return l_sim(Se, Sl, M, gamma, rho), t, M


def grad_latent(X: np.ndarray, L: np.ndarray, gamma: float = 0.6, q: float = 0.005) -> np.ndarray:
    """dL_sim / dL with the mask held fixed (it is piecewise constant in the
    latents): for each masked pair the derivative of its squared residual,
    2 r_ij (l_i - l_j) / S_lat(i, j) toward l_i, summed over both orders
    (the sum runs over ordered pairs), divided by sum(Mask). Pairs at zero
    latent distance contribute nothing."""
    X = np.asarray(X, np.float64)
    L = np.asarray(L, np.float64)
    rho = math.sqrt(L.shape[1] / X.shape[1])
    Se, Sl = pairwise_l2(X), pairwise_l2(L)
    M = mask(Se, Sl, tau_emb(Se, q), gamma, rho)
    G = np.zeros_like(L)
    n = M.sum()
    B = L.shape[0]
    for i in range(B):
        for j in range(B):
            if not M[i, j] or Sl[i, j] == 0.0:
                continue
            r = Sl[i, j] - gamma * rho * Se[i, j]
            u = (L[i] - L[j]) / Sl[i, j]
            G[i] += 2.0 * r * u / n   # from the term (i, j)
            G[j] -= 2.0 * r * u / n   # the same term through l_j
    return G

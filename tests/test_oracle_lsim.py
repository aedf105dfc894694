"""The oracle's selective similarity loss (Sec. 3.2.2, Eq. "similarityconfig"
and "equation8"; tau_emb per Sec. 4.5.1), pinned by hand-worked batches, a
closed form and finite differences."""
import math

import numpy as np
import pytest

from oracle import lsim


def test_hand_worked_batch():
    """Four embeddings on a line at 0, 1, 3, 7 (E_dim = 1) and latents at
    0, 2, 2, 9 (L_dim = 1): rho = 1, gamma = 0.5. Unordered pairs and their
    distances (emb, lat): (0,1) 1,2; (0,2) 3,2; (0,3) 7,9; (1,2) 2,0;
    (1,3) 6,7; (2,3) 4,7. With 6 pairs, q = 0.2 gives position
    ceil(1.2) - 1 = 1 of the sorted embedding distances 1,2,3,4,6,7: tau = 2.
    Mask: S_emb <= 2 (pairs (0,1), (1,2)) or S_lat <= gamma rho tau = 1
    (pair (1,2)): pairs (0,1) and (1,2), both orders, 4 entries.
    Residuals S_lat - 0.5 S_emb: (0,1) 2 - 0.5 = 1.5, (1,2) 0 - 1 = -1.
    L_sim = 2 (1.5^2 + 1^2) / 4 = 1.625."""
    X = np.array([[0.0], [1.0], [3.0], [7.0]])
    L = np.array([[0.0], [2.0], [2.0], [9.0]])
    loss, tau, M = lsim.batch_loss(X, L, gamma=0.5, q=0.2)
    assert tau == 2.0
    want = np.zeros((4, 4), bool)
    for i, j in [(0, 1), (1, 2)]:
        want[i, j] = want[j, i] = True
    assert np.array_equal(M, want)
    assert loss == 1.625


def test_latent_threshold_adds_pairs():
    """The second condition of the mask: a pair far apart in the embedding
    space but close in the latent space is included (the anti-collapse
    term). Embeddings 0, 10, 20; latents 0, 0.1, 50; gamma rho tau = 0.6 * 1 *
    10 = 6 with q = 0.1 (3 pairs: position 0, the smallest distance 10):
    pairs with S_emb <= 10: (0,1), (1,2); with S_lat <= 6: (0,1). Residuals
    (0,1) 0.1 - 6 = -5.9, (1,2) 49.9 - 6 = 43.9; loss = (5.9^2 + 43.9^2) / 2."""
    X = np.array([[0.0], [10.0], [20.0]])
    L = np.array([[0.0], [0.1], [50.0]])
    loss, tau, M = lsim.batch_loss(X, L, gamma=0.6, q=0.1)
    assert tau == 10.0
    assert M.sum() == 4 and M[0, 1] and M[1, 2] and not M[0, 2]
    assert loss == pytest.approx((5.9 ** 2 + 43.9 ** 2) / 2, rel=1e-14)
    # far in both spaces: not masked
    L2 = np.array([[0.0], [30.0], [90.0]])
    _, _, M2 = lsim.batch_loss(X, L2, gamma=0.6, q=0.1)
    assert M2.sum() == 4 and M2[0, 1] and M2[1, 2]


def test_scaled_copy_has_zero_loss():
    """Latents that are the embeddings scaled by gamma rho (and rotated)
    reproduce S_lat = gamma rho S_emb on every pair: L_sim = 0."""
    rng = np.random.default_rng(1)
    X = rng.normal(size=(64, 8))
    Q, _ = np.linalg.qr(rng.normal(size=(8, 8)))
    gamma = 0.6
    rho = math.sqrt(8 / 8)
    L = gamma * rho * X @ Q
    loss, _, M = lsim.batch_loss(X, L, gamma=gamma)
    assert M.sum() > 0 and loss == pytest.approx(0.0, abs=1e-24)


def test_tau_selects_the_closest_half_percent():
    rng = np.random.default_rng(2)
    X = rng.normal(size=(300, 16))
    S = lsim.pairwise_l2(X)
    t = lsim.tau_emb(S)
    iu = np.triu_indices(300, 1)
    n = (S[iu] <= t).sum()
    assert n == math.ceil(0.005 * iu[0].size)  # continuous data: no ties
    # the definition of S: against a direct distance
    assert S[3, 7] == pytest.approx(np.sqrt(((X[3] - X[7]) ** 2).sum()), rel=1e-15)


def test_gradient_matches_finite_differences():
    """grad_latent against central differences of the loss with the mask
    held fixed (batches where no pair sits on a mask boundary)."""
    rng = np.random.default_rng(3)
    X = rng.normal(size=(40, 6))
    L = rng.normal(size=(40, 3))
    gamma = 0.6
    rho = math.sqrt(3 / 6)
    Se = lsim.pairwise_l2(X)
    t = lsim.tau_emb(Se)
    M = lsim.mask(Se, lsim.pairwise_l2(L), t, gamma, rho)
    G = lsim.grad_latent(X, L, gamma)
    h = 1e-6
    for i, k in [(0, 0), (5, 1), (17, 2), (39, 0)]:
        Lp, Lm = L.copy(), L.copy()
        Lp[i, k] += h
        Lm[i, k] -= h
        fp = lsim.l_sim(Se, lsim.pairwise_l2(Lp), M, gamma, rho)
        fm = lsim.l_sim(Se, lsim.pairwise_l2(Lm), M, gamma, rho)
        assert G[i, k] == pytest.approx((fp - fm) / (2 * h), rel=1e-5, abs=1e-9)

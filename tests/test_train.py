"""The package's encoder training (Sec. 3.2.2, Sec. 4.5.1) against the
oracle's statement of L_sim, the BatchNorm folding, and a short CPU run."""
import math

import numpy as np
import pytest

from oracle import lsim


def _torch():
    return pytest.importorskip("torch")


@pytest.mark.parametrize("B,E,L", [(40, 8, 3), (200, 16, 4), (97, 128, 24)])
def test_loss_and_gradient_equal_the_oracle(B, E, L):
    torch = _torch()
    from paper_2608_15438_gb300 import train

    rng = np.random.default_rng(B)
    X = rng.normal(size=(B, E))
    Z = rng.normal(size=(B, L))
    loss_o, tau_o, M_o = lsim.batch_loss(X, Z, gamma=0.6)
    G_o = lsim.grad_latent(X, Z, gamma=0.6)
    Xt = torch.tensor(X, dtype=torch.float64)
    Zt = torch.tensor(Z, dtype=torch.float64, requires_grad=True)
    loss, tau, nm = train.lsim_loss(torch, Xt, Zt, gamma=0.6, eps=1e-30)
    loss.backward()
    assert float(tau) == pytest.approx(tau_o, rel=1e-12)
    assert int(nm) == int(M_o.sum())
    assert loss.item() == pytest.approx(loss_o, rel=1e-10)
    assert np.allclose(Zt.grad.numpy(), G_o, rtol=1e-8, atol=1e-12)


def test_batchnorm_folds_into_the_linear_layers():
    torch = _torch()
    from paper_2608_15438_gb300 import train

    torch.manual_seed(0)
    model = train.make_encoder(torch, 16, (32, 8), 4).double()
    x = torch.randn(256, 16, dtype=torch.float64)
    model.train()
    for _ in range(5):  # move the running statistics away from 0 / 1
        model(x * 3 + 1)
    for m in model:
        if isinstance(m, torch.nn.BatchNorm1d):
            m.weight.data.uniform_(0.5, 2.0)
            m.bias.data.uniform_(-1, 1)
    model.eval()
    want = model(x).detach().numpy()
    layers = train.fold_batchnorm(torch, model)
    assert [W.shape for W, _ in layers] == [(32, 16), (8, 32), (4, 8)]
    h = x.numpy()
    for i, (W, b) in enumerate(layers):
        h = h @ W.astype(np.float64).T + b
        if i + 1 < len(layers):
            h = np.maximum(h, 0.0)
    assert np.allclose(h, want, rtol=1e-5, atol=1e-5)
    w = train.index_weights(layers)
    assert len(w) == 5 and len(w[4]) == 1 and w[2].shape == (4, 8)


def test_short_training_lowers_the_loss(tmp_path):
    torch = _torch()
    import synth
    from paper_2608_15438_gb300 import train

    w = synth.WORKLOADS["tiny"]
    x = torch.from_numpy(synth.base(w, 4096))
    hist = []
    weights, h = train.train_encoder(torch, x, w.in_scale, (64,), 8, epochs=6, batch=512, lr=2e-3,
                                     log=hist.append)
    assert len(h) == 6 and h[-1][1] < h[0][1]
    assert weights[0].shape == (64, 128) and weights[2].shape == (8, 64)
    path = str(tmp_path / "enc.npz")
    train.save_weights(path, weights, h)
    back = train.load_weights(path)
    assert all(np.array_equal(a, b) for a, b in zip(back, weights))

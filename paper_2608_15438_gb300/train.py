"""Encoder training with the selective similarity-preservation loss.

The encoder E maps an embedding to L_dim latent logits (Sec. 3.2.1); it is
trained so that pairwise Euclidean distances among near neighbours survive
the map (Sec. 3.2.2): for a mini-batch of B vectors with distance matrices
S_emb (embeddings) and S_lat (latents), rho = sqrt(L_dim / E_dim) and a scale
gamma,
    Mask(i, j) = [i != j and (S_emb(i, j) <= tau_emb or S_lat(i, j) <= gamma rho tau_emb)]
    L_sim = sum_ij Mask(i, j) (S_lat(i, j) - gamma rho S_emb(i, j))^2 / sum(Mask)
with tau_emb set in every mini-batch so that the closest 0.5% of its pairs
fall within it (Sec. 4.5.1). The protocol of Sec. 4.5.1: a fixed subset of
the base, mini-batches of 4096, Adam at 2e-4, gamma = 0.6. Hidden layers are
Linear -> BatchNorm -> ReLU and the last layer is linear (Sec. 4.5.1, Table
"NeuRoute-arch"); at export each BatchNorm (an affine map at inference) is
folded into its Linear, giving the index format's W1, b1, middle layers, W2,
b2.

This runs off the query path, once per index: PyTorch autograd and Adam do
the optimisation on the GPU, and the weights it returns are the index's data
(the query path's kernels then run the encoder forward). uint8 embeddings are
scaled by in_scale (1/255) for training, as the index's encoder scales them.
"""
from __future__ import annotations

import math
import time

import numpy as np


def make_encoder(torch, D: int, widths, b: int):
    """Linear -> BatchNorm1d -> ReLU for each hidden width, then Linear(b)."""
    nn = torch.nn
    layers, prev = [], D
    for w in widths:
        layers += [nn.Linear(prev, w), nn.BatchNorm1d(w), nn.ReLU()]
        prev = w
    layers.append(nn.Linear(prev, b))
    return nn.Sequential(*layers)


def pairwise_l2(torch, Z, eps: float = 0.0):
    """S(i, j) = ||z_i - z_j||_2 from the Gram matrix, clamped at eps before the
    square root (eps > 0 keeps the gradient finite for coincident points)."""
    n = (Z * Z).sum(1)
    sq = n[:, None] + n[None, :] - 2.0 * (Z @ Z.T)
    return torch.sqrt(torch.clamp(sq, min=eps))


def lsim_loss(torch, X, Z, gamma: float = 0.6, q: float = 0.005, eps: float = 1e-12):
    """L_sim of one mini-batch: embeddings X [B x E_dim] (no gradient), latents
    Z [B x L_dim]; returns (loss, tau_emb, sum(Mask)). tau_emb is the distance
    of the ceil(q B (B - 1) / 2)-th closest unordered pair of the batch."""
    B = X.shape[0]
    rho = math.sqrt(Z.shape[1] / X.shape[1])
    with torch.no_grad():
        Se = pairwise_l2(torch, X)
        # the k-th smallest of the B (B - 1) / 2 pairs i < j: sorting the
        # strict upper triangle with zeros elsewhere puts the B (B + 1) / 2
        # zeros first (distances are non-negative, so ties with zero pairs
        # change no value)
        k = max(1, math.ceil(q * (B * (B - 1) // 2)))
        tau = torch.sort(torch.triu(Se, diagonal=1).reshape(-1)).values[B * (B + 1) // 2 + k - 1]
    Sl = pairwise_l2(torch, Z, eps)
    M = (Se <= tau) | (Sl.detach() <= gamma * rho * tau)
    M.fill_diagonal_(False)
    r = Sl - gamma * rho * Se
    nm = M.sum()
    return (r * r * M).sum() / nm, tau, nm


def fold_batchnorm(torch, model):
    """Weights of the trained encoder in the index's form: a list of (W, b) per
    linear layer, each hidden layer's BatchNorm (running statistics) folded
    in: W' = diag(g / sqrt(var + e)) W, b' = (b - mean) g / sqrt(var + e) + beta."""
    mods = list(model)
    out = []
    i = 0
    while i < len(mods):
        lin = mods[i]
        W = lin.weight.detach().double()
        bb = lin.bias.detach().double()
        if i + 1 < len(mods) and isinstance(mods[i + 1], torch.nn.BatchNorm1d):
            bn = mods[i + 1]
            s = bn.weight.detach().double() / torch.sqrt(bn.running_var.double() + bn.eps)
            W = W * s[:, None]
            bb = (bb - bn.running_mean.double()) * s + bn.bias.detach().double()
            i += 3  # Linear, BatchNorm, ReLU
        else:
            i += 1
        out.append((W.float().cpu().numpy(), bb.float().cpu().numpy()))
    return out


def index_weights(layers):
    """(W1, b1, W2, b2) or (W1, b1, W2, b2, ((W, b), ...)) as the index
    builders take them, from the folded layers."""
    (W1, b1), (W2, b2) = layers[0], layers[-1]
    mid = tuple(layers[1:-1])
    return (W1, b1, W2, b2) + ((mid,) if mid else ())


def train_encoder(torch, x, in_scale: float, widths, b: int, epochs: int = 500, batch: int = 4096,
                  lr: float = 2e-4, gamma: float = 0.6, q: float = 0.005, seed: int = 0, log=None):
    """Train on the rows x [n x D] (a device tensor, uint8 or fp32); returns
    (index weights, history), history one (epoch, mean loss, mean tau_emb,
    seconds) per epoch."""
    dev = x.device
    torch.manual_seed(seed)
    model = make_encoder(torch, x.shape[1], widths, b).to(dev)
    opt = torch.optim.Adam(model.parameters(), lr=lr)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    n = x.shape[0]
    hist = []
    t0 = time.time()
    for ep in range(epochs):
        model.train()
        perm = torch.randperm(n, device=dev, generator=g)
        tot, ttot, nb = torch.zeros((), device=dev), torch.zeros((), device=dev), 0
        for s in range(0, n - batch + 1, batch):
            xb = x[perm[s:s + batch]].float() * in_scale
            loss, tau, _ = lsim_loss(torch, xb, model(xb), gamma, q)
            opt.zero_grad(set_to_none=True)
            loss.backward()
            opt.step()
            tot += loss.detach()
            ttot += tau
            nb += 1
        hist.append((ep, float(tot) / max(nb, 1), float(ttot) / max(nb, 1), time.time() - t0))
        if log is not None:
            log(hist[-1])
    model.eval()
    return index_weights(fold_batchnorm(torch, model)), hist


def save_weights(path: str, weights, history=None, meta=None):
    """Write index weights (and the training history) to an .npz file."""
    arrs = {"W1": weights[0], "b1": weights[1], "W2": weights[2], "b2": weights[3]}
    for i, (W, bb) in enumerate(weights[4] if len(weights) > 4 else ()):
        arrs[f"Wm{i}"], arrs[f"bm{i}"] = W, bb
    if history is not None:
        arrs["history"] = np.asarray(history, np.float64)
    if meta is not None:
        arrs["meta"] = np.frombuffer(repr(meta).encode(), np.uint8)
    np.savez(path, **arrs)


def load_weights(path: str):
    """Index weights from save_weights' file."""
    z = np.load(path)
    mid, i = [], 0
    while f"Wm{i}" in z:
        mid.append((z[f"Wm{i}"], z[f"bm{i}"]))
        i += 1
    out = (z["W1"], z["b1"], z["W2"], z["b2"])
    return out + ((tuple(mid),) if mid else ())


def main():
    """python -m paper_2608_15438_gb300.train --workload u8-100m --out enc.npz
    trains the workload's encoder shape on the first --rows base rows."""
    import argparse
    import json
    import os
    import sys

    import torch

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    import synth

    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="u8-100m")
    ap.add_argument("--rows", type=int, default=2_000_000)
    ap.add_argument("--epochs", type=int, default=500)
    ap.add_argument("--batch", type=int, default=4096)
    ap.add_argument("--lr", type=float, default=2e-4)
    ap.add_argument("--gamma", type=float, default=0.6)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--out", required=True)
    a = ap.parse_args()
    w = synth.WORKLOADS[a.workload]
    dev = torch.device("cuda", 0)
    x = synth.DeviceRows(w, synth.SEED_DATA, device=0).rows(0, min(a.rows, w.n))
    widths = (w.hidden,) + tuple(w.mid)
    weights, hist = train_encoder(torch, x, w.in_scale, widths, w.bits, a.epochs, a.batch, a.lr,
                                  a.gamma, seed=a.seed,
                                  log=lambda h: print(json.dumps({"epoch": h[0], "loss": h[1],
                                                                  "tau_emb": h[2], "s": h[3]}),
                                                      flush=True))
    save_weights(a.out, weights, hist, {"workload": a.workload, "rows": a.rows, "epochs": a.epochs,
                                        "batch": a.batch, "lr": a.lr, "gamma": a.gamma})


if __name__ == "__main__":
    main()

"""Encoder training on the GPU (Sec. 3.2.2, protocol Sec. 4.5.1): a short run
lowers L_sim, the GPU loss of a batch agrees with the oracle's, and an index
built from the trained (BatchNorm-folded, biased) weights is searched by the
GPU exactly as by the oracle."""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import need_cuda
from oracle import lsim

pytestmark = pytest.mark.gpu


def test_training_on_gpu_and_an_index_from_its_weights(tmp_path):
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr
    from paper_2608_15438_gb300 import train
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    dev = torch.device("cuda", 0)
    x = synth.DeviceRows(w, synth.SEED_DATA, device=0).rows(0, 16384)
    weights, hist = train.train_encoder(torch, x, w.in_scale, (256,), 12, epochs=5, batch=2048,
                                        lr=2e-3, seed=1)
    assert hist[-1][1] < hist[0][1]
    # one batch's loss in fp32 on the GPU against the oracle's float64 value
    xb = x[:512].float() * w.in_scale
    model = train.make_encoder(torch, 128, (256,), 12).to(dev)
    with torch.no_grad():
        zb = model(xb)
        loss, tau, nm = train.lsim_loss(torch, xb, zb)
    lo, to, Mo = lsim.batch_loss(xb.double().cpu().numpy(), zb.double().cpu().numpy())
    assert float(tau) == pytest.approx(to, rel=1e-5)
    assert abs(int(nm) - int(Mo.sum())) <= 4  # at most a pair on either threshold moves
    assert float(loss) == pytest.approx(lo, rel=1e-3)
    # the trained weights are index data: build, then search on the GPU and in the oracle
    assert np.any(weights[1] != 0) and np.any(weights[3] != 0)
    base = synth.base(w, 20000)
    path = str(tmp_path / "trained.nrix")
    build_index(config(w.dtype, w.dim, 256, 12, w.k_max, w.t), base, weights, path)
    ix = nr.Index(path, 0)
    orc = oracle.Index(path)
    qs = synth.queries(w, 200)
    lg = orc.encode(qs)
    dq = torch.from_numpy(qs).cuda()
    lg_gpu = ix.encode(dq).cpu().numpy()
    err = np.abs(lg_gpu - lg).max(1) / np.abs(lg).max(1)
    assert err.max() <= 1e-2
    ids, d = ix.search_logits(dq, torch.from_numpy(lg).cuda(), 10, 32, 64)
    torch.cuda.synchronize()
    ids_o, d_o, _ = orc.search(qs, 10, 32, 64, oracle.params(), logits=lg)
    assert np.array_equal(ids.cpu().numpy(), ids_o) and np.array_equal(d.cpu().numpy(), d_o)
    ix.close()

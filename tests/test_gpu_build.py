"""GPU index construction (neuroute_build.h) against the host builder: fed the
same logits, both must write the same bytes (thresholds, codes, clusters,
centroids, ids, rows). Cases cover one warp per bucket and one CTA per large
bucket, K = 1 and K > 1, seeding with all-zero weights, small samples, chunked
passes in any order, and the call-order and input errors. A GPU-encoded build
is then searched and checked against the oracle on its saved file."""
import os

import numpy as np
import pytest

import oracle
import synth
from gpu_util import need_cuda, recall
from nrix_reader import read_nrix
from paper_2608_15438_gb300.builder import build_index_from_logits, config, encode

pytestmark = pytest.mark.gpu


def gpu_build(torch, cfg, base, logits, weights, chunks=1, order=None):
    from paper_2608_15438_gb300 import neuroute as nr

    N = base.shape[0]
    bd = nr.Builder(cfg, N, weights, 0)
    cuts = np.linspace(0, N, chunks + 1).astype(np.int64)
    ranges = list(zip(cuts[:-1], cuts[1:]))
    order = order or list(range(len(ranges)))
    for i in order:
        a, b = ranges[i]
        if logits is None:
            bd.encode(torch.from_numpy(base[a:b]).cuda(), int(a))
        else:
            bd.set_logits(torch.from_numpy(logits[a:b]).cuda(), int(a))
    torch.cuda.synchronize()
    info = bd.finish()
    for i in reversed(order):
        a, b = ranges[i]
        bd.place(torch.from_numpy(base[a:b]).cuda(), int(a))
    ix = bd.end()
    return ix, info


def same_as_host(tmp_path, torch, cfg, base, logits, weights, **kw):
    ph = str(tmp_path / "host.nrix")
    info_h = build_index_from_logits(cfg, base, logits, weights, ph)
    ix, info_g = gpu_build(torch, cfg, base, logits, weights, **kw)
    pg = str(tmp_path / "gpu.nrix")
    ix.save(pg)
    ix.close()
    a, g = read_nrix(ph), read_nrix(pg)
    for name in ("tau", "bkt_off", "cl_off", "cent", "ids", "vec"):
        assert np.array_equal(a[name], g[name]), name
    assert open(ph, "rb").read() == open(pg, "rb").read()
    assert info_h == info_g
    return info_g


def tiny_inputs(n, b):
    w = synth.WORKLOADS["tiny"]
    base = synth.base(w, n)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    return w, base, (W1, b1, W2[:b], b2[:b])


@pytest.mark.parametrize("n,b,kmax,t,spc,chunks", [
    (100_000, 16, 4, 32, 256, 1),    # the tiny workload's index: warp buckets, K up to 4
    (60_000, 6, 8, 8, 256, 3),       # ~940 rows a bucket, K = 8 on warps, passes in 3 chunks
    (40_000, 2, 16, 64, 256, 2),     # 10,000-row buckets: one CTA each, K = 16
    (50_000, 3, 1, 64, 256, 1),      # no clustering: CTA buckets with K = 1
    (30_000, 4, 16, 4, 3, 1),        # sample of 3 per cluster: strided sample m < n
])
def test_same_bytes_as_host_builder(tmp_path, n, b, kmax, t, spc, chunks):
    torch = need_cuda()
    w, base, weights = tiny_inputs(n, b)
    cfg = config(w.dtype, w.dim, w.hidden, b, kmax, t, sample_per_cluster=spc)
    logits = encode(cfg, base, weights)
    order = list(range(chunks))[::-1] if chunks > 1 else None
    info = same_as_host(tmp_path, torch, cfg, base, logits, weights, chunks=chunks, order=order)
    assert info["n_clusters"] >= info["n_buckets"]


def test_degenerate_inputs(tmp_path):
    """N = 1; all rows with equal logits (every seeding weight is zero, every
    distance ties); a single distinct value per column."""
    torch = need_cuda()
    w, base, weights = tiny_inputs(5000, 8)
    cfg = config(w.dtype, w.dim, w.hidden, 8, 8, 16)
    same_as_host(tmp_path, torch, cfg, base[:1], encode(cfg, base[:1], weights), weights)
    flat = np.tile(np.linspace(-1, 1, 8, dtype=np.float32), (5000, 1))
    info = same_as_host(tmp_path, torch, cfg, base, flat, weights)
    assert info["n_buckets"] == 1 and info["n_clusters"] == 1   # one bucket; empties dropped
    two = np.where(np.arange(5000)[:, None] % 2 == 0, 1.0, -1.0).astype(np.float32) * np.ones((1, 8), np.float32)
    same_as_host(tmp_path, torch, cfg, base, two, weights)


def test_gpu_encoded_build_searches_like_the_oracle(tmp_path):
    """The GPU's own encoder builds the index; its saved file, loaded by the
    oracle, gives the same results as the in-memory index."""
    torch = need_cuda()
    w, base, weights = tiny_inputs(100_000, 16)
    cfg = config(w.dtype, w.dim, w.hidden, 16, w.k_max, w.t)
    ix, info = gpu_build(torch, cfg, base, None, weights, chunks=4)
    path = str(tmp_path / "enc.nrix")
    ix.save(path)
    orc = oracle.Index(path)
    qs = synth.queries(w, 500)
    lg = orc.encode(qs)
    kw = dict(t_low=4)
    ix.set_params(**kw)
    ids, d = ix.search_logits(torch.from_numpy(qs).cuda(), torch.from_numpy(lg).cuda(), 10, 16, 64)
    torch.cuda.synchronize()
    ids_o, d_o, _ = orc.search(qs, 10, 16, 64, oracle.params(**kw), logits=lg)
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    truth = oracle.bruteforce(base, qs, 10)[0]
    assert recall(ids_o, truth) > 0.5
    # tau: exact lower medians of the GPU encoder's logits, which agree with
    # the host's fp32 encoder to within fp16 rounding
    tau_host = np.sort(encode(cfg, base, weights), axis=0)[(base.shape[0] - 1) // 2]
    assert np.allclose(read_nrix(path)["tau"], tau_host, atol=2e-2)
    ix.close()


def test_call_order_and_input_errors():
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr

    w, base, weights = tiny_inputs(1000, 8)
    cfg = config(w.dtype, w.dim, w.hidden, 8, 4, 16)
    lg = torch.from_numpy(encode(cfg, base, weights)).cuda()
    rows = torch.from_numpy(base).cuda()
    bd = nr.Builder(cfg, 1000, weights, 0)
    with pytest.raises(nr.NRError):
        bd.place(rows, 0)                      # before finish
    bd.set_logits(lg[:500], 0)
    with pytest.raises(nr.NRError):
        bd.finish()                            # rows 500.. have no logits
    with pytest.raises(nr.NRError):
        bd.set_logits(lg[:600], 500)           # past N
    bd.set_logits(lg[500:], 500)
    torch.cuda.synchronize()
    bd.finish()
    with pytest.raises(nr.NRError):
        bd.set_logits(lg, 0)                   # pass 1 is over
    bd.place(rows[:999], 0)
    with pytest.raises(nr.NRError):
        bd.end()                               # one row never placed; frees the build
    bad = lg.clone()
    bad[7, 3] = float("nan")
    bd = nr.Builder(cfg, 1000, weights, 0)
    bd.set_logits(bad, 0)
    torch.cuda.synchronize()
    with pytest.raises(nr.NRError):
        bd.finish()
    bd.close()
    for kw in (dict(K_max=65), dict(b=25), dict(t=0)):
        c = config(w.dtype, w.dim, w.hidden, 8, 4, 16)
        for k, v in kw.items():
            setattr(c, k, v)
        with pytest.raises(nr.NRError):
            nr.Builder(c, 1000, weights, 0)


def test_extract_gives_the_same_results(tmp_path):
    """A sub-index of the buckets some queries probe: the oracle on it gives
    those queries exactly the ids, distances and statistics the GPU gives on
    the whole index."""
    torch = need_cuda()
    w, base, weights = tiny_inputs(100_000, 16)
    cfg = config(w.dtype, w.dim, w.hidden, 16, w.k_max, w.t)
    ix, _ = gpu_build(torch, cfg, base, None, weights)
    qs = synth.queries(w, 64)
    dq = torch.from_numpy(qs).cuda()
    lg = ix.encode(dq)
    P, C, kw = 32, 64, dict(t_low=2)
    codes, nprobe = ix.route(lg, P)
    ix.set_params(**kw)
    ids, d = ix.search_logits(dq, lg, 10, P, C)
    st = ix.query_stats(64)
    torch.cuda.synchronize()
    c = codes.cpu().numpy().view(np.uint32)
    used = np.concatenate([c[i, :n] for i, n in enumerate(nprobe.cpu().numpy())])
    sub = str(tmp_path / "sub.nrix")
    rows, ncl = ix.extract(used, sub)
    assert 0 < rows < base.shape[0] and 0 < ncl < ix.n_clusters
    orc = oracle.Index(sub)
    ids_o, d_o, st_o = orc.search(qs, 10, P, C, oracle.params(**kw), logits=lg.cpu().numpy())
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)
    from paper_2608_15438_gb300 import neuroute as nr
    with pytest.raises(nr.NRError):
        ix.extract(np.array([1 << 16], np.uint32), sub)   # code out of range
    ix.close()

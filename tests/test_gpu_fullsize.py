"""Parity at the benchmark's full sizes and launch configuration: 1e7-vector
workloads, the whole 10,000-query batch in one nr_search_logits call with the
benchmark's (P, C, t_low), checked against the oracle on a sample of queries
spread over the batch (the oracle computes each one from scratch).

Fed the oracle's logits, ids, distances and per-query statistics must match
exactly; end to end (GPU encoder), Recall@10 on the sample must agree with the
oracle's within 0.002 against brute-force ground truth."""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import cached_index, need_cuda, recall

pytestmark = pytest.mark.gpu

SAMPLE = 200


@pytest.mark.parametrize("name", ["u8-10m", "f32-10m"])
def test_full_batch_sampled_parity(name):
    torch = need_cuda()
    import bench
    from paper_2608_15438_gb300 import neuroute as nr

    w = synth.WORKLOADS[name]
    op = bench.OPERATING_POINTS[name]
    P, C = op["P"], op["C"]
    path = cached_index(name)
    ix = nr.Index(path, 0)
    kw = bench.op_params(w, ix)
    orc = oracle.Index(path)
    qs = synth.queries(w)
    lg = orc.encode(qs)
    dq = torch.from_numpy(qs).cuda()
    ix.set_params(**kw)
    ids, d = ix.search_logits(dq, torch.from_numpy(lg).cuda(), 10, P, C)
    st = ix.query_stats(w.nq)
    torch.cuda.synchronize()
    ids, d, st = ids.cpu().numpy(), d.cpu().numpy(), st.cpu().numpy()
    sample = np.linspace(0, w.nq - 1, SAMPLE).astype(np.int64)
    p = oracle.params(**bench.method_kw(kw))
    ids_o, d_o, st_o = orc.search(qs[sample], 10, P, C, p, logits=lg[sample])
    assert np.array_equal(ids[sample], ids_o)
    if w.dtype == "u8":
        assert np.array_equal(d[sample], d_o)
    else:
        assert np.all(np.abs(d[sample] - d_o) <= 1e-5 * np.abs(d_o))
    assert np.array_equal(st[sample], st_o)
    # end to end through the GPU encoder, recall against exact k-NN on the sample
    ids_e, _ = ix.search(dq, 10, P, C)
    torch.cuda.synchronize()
    ids_oe, _, _ = orc.search(qs[sample], 10, P, C, p)
    base = torch.from_numpy(synth.base(w)).cuda().float()
    qf = dq[torch.from_numpy(sample).cuda()].float()
    dist = (qf * qf).sum(1, keepdim=True) + (base * base).sum(1)[None] - 2.0 * qf @ base.T
    truth = torch.topk(dist, 10, dim=1, largest=False).indices.cpu().numpy()
    del base, dist
    r_gpu = recall(ids_e.cpu().numpy()[sample], truth)
    r_orc = recall(ids_oe, truth)
    assert abs(r_gpu - r_orc) <= 0.002 + 1e-12, (r_gpu, r_orc)
    ix.close()


@pytest.mark.parametrize("name,sample_n", [("u8-100m", 200), ("u8-1b", 100)])
def test_gpu_built_sampled_parity(name, sample_n):
    """1e8 and 1e9 uint8 vectors, index built on the GPU, the whole
    10,000-query batch in one nr_search_logits call at the benchmark's
    operating point; sample_n sampled queries checked against the oracle,
    which answers them from the sub-index of the buckets its own probe lists
    name (its own logits too). End to end (GPU encoder), Recall@10 on the
    sample agrees with the oracle's within 0.002 against exact k-NN."""
    torch = need_cuda()
    import os
    import tempfile

    import bench
    from paper_2608_15438_gb300 import neuroute as nr

    torch.cuda.empty_cache()
    w = synth.WORKLOADS[name]
    op = bench.OPERATING_POINTS[name]
    P, C = op["P"], op["C"]
    dev = torch.device("cuda", 0)
    ix, _ = bench.gpu_index(w, torch, nr, dev)
    kw = bench.op_params(w, ix)       # a calibrated gate and S_max are fitted on this index
    qs = synth.queries(w)
    lg = oracle.encode_weights(synth.encoder_weights(w), w.in_scale, qs)
    dq = torch.from_numpy(qs).cuda()
    ix.set_params(**kw)
    ids, d = ix.search_logits(dq, torch.from_numpy(lg).cuda(), 10, P, C)
    st = ix.query_stats(w.nq)
    torch.cuda.synchronize()
    ids, d, st = ids.cpu().numpy(), d.cpu().numpy(), st.cpu().numpy()
    sample = np.linspace(0, w.nq - 1, sample_n).astype(np.int64)
    p = oracle.params(**bench.method_kw(kw))
    with tempfile.TemporaryDirectory() as td:
        sub = os.path.join(td, "sub.nrix")
        bench.oracle_subindex(w, ix, qs[sample], P, kw, sub)
        orc = oracle.Index(sub)
        ids_o, d_o, st_o = orc.search(qs[sample], 10, P, C, p, logits=lg[sample])
        assert np.array_equal(ids[sample], ids_o)
        assert np.array_equal(d[sample], d_o)
        assert np.array_equal(st[sample], st_o)
        ids_oe, _, _ = orc.search(qs[sample], 10, P, C, p)
        orc.close()
    ids_e, _ = ix.search(dq, 10, P, C)
    torch.cuda.synchronize()
    truth = bench.ground_truth_rows(torch, w, dq[torch.from_numpy(sample).cuda()], 10, dev)
    r_gpu = recall(ids_e.cpu().numpy()[sample], truth)
    r_orc = recall(ids_oe, truth)
    assert abs(r_gpu - r_orc) <= 0.002 + 1e-12, (r_gpu, r_orc)
    ix.close()
    del ix
    torch.cuda.empty_cache()


def test_ground_truth_1e8_against_oracle_bruteforce():
    """The benchmark's ground truth over 1e8 uint8 rows regenerated on the GPU
    (bench.ground_truth_rows: TF32 matmul, exact for uint8, with the group
    pre-selection) equals the oracle's brute-force k-NN on 200 queries: the
    oracle scans the same rows drawn by the host generator, chunk by chunk,
    and the chunks' exact top-k lists are merged by (distance, id)."""
    torch = need_cuda()
    import bench

    w = synth.WORKLOADS["u8-100m"]
    k, nq = 10, 200
    qs = synth.queries(w, nq)
    dev = torch.device("cuda", 0)
    got = bench.ground_truth_rows(torch, w, torch.from_numpy(qs).to(dev), k, dev)
    best_i = np.full((nq, k), -1, np.int64)
    best_d = np.full((nq, k), np.inf)
    got_d = np.full((nq, k), -1, np.int64)
    chunk = 10_000_000
    for r0 in range(0, w.n, chunk):
        m = min(chunk, w.n - r0)
        X = synth.mixture(w, synth.SEED_DATA, r0, m)
        ci, cd = oracle.bruteforce(X, qs, k)
        ai = np.concatenate([best_i, ci + r0], 1)
        ad = np.concatenate([best_d, cd.astype(np.float64)], 1)
        for qi in range(nq):
            o = np.lexsort((ai[qi], ad[qi]))[:k]
            best_i[qi], best_d[qi] = ai[qi][o], ad[qi][o]
        # the distance of each GPU-found id, from the rows of this chunk
        inside = (got >= r0) & (got < r0 + m)
        if inside.any():
            qq, kk = np.nonzero(inside)
            rows = X[got[qq, kk] - r0].astype(np.int64)
            got_d[qq, kk] = ((rows - qs[qq].astype(np.int64)) ** 2).sum(1)
        del X
    assert np.all(got_d >= 0)
    # the same distances at every rank (ids may differ only among equal distances)
    assert np.array_equal(np.sort(got_d, 1), best_d.astype(np.int64))

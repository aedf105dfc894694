"""The pipelined search (pipe_chunk > 0: refinement of one chunk on a library
stream overlapping route and select of the next ones, three chunk buffers)
and the refinement block cap give exactly the results, statistics and kernel
sequence of the plain search: chunk sizes that divide the batch or not, one
query per chunk, more chunks than buffers, caps from 1 block per SM; timing
still reports every stage; the caller's stream sees the results."""
import numpy as np
import pytest

import synth
from gpu_util import build_small, need_cuda

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return need_cuda()


@pytest.fixture(scope="module")
def tiny(torch, tmp_path_factory):
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, _ = build_small(tmp_path_factory.mktemp("pipe"), "tiny", n=100_000, bits=16)
    w = synth.WORKLOADS["tiny"]
    qs = synth.queries(w, 1000)
    return {"ix": nr.Index(path, 0), "dq": torch.from_numpy(qs).cuda()}


BASE = dict(t_low=4, gate_m0=0.0, gate_m1=2.0)


def run(tiny, torch, stream=None, **kw):
    ix = tiny["ix"]
    ix.set_params(**{**BASE, **kw})
    try:
        ids, d = ix.search(tiny["dq"], 10, 64, 128, stream=stream)
        st = ix.query_stats(tiny["dq"].shape[0])
        torch.cuda.synchronize()
    finally:
        ix.set_params()
    return ids.cpu().numpy(), d.cpu().numpy(), st.cpu().numpy()


@pytest.mark.parametrize("kw", [dict(pipe_chunk=1000), dict(pipe_chunk=999), dict(pipe_chunk=250),
                                dict(pipe_chunk=77), dict(pipe_chunk=1), dict(refine_ctas=1),
                                dict(refine_ctas=3), dict(pipe_chunk=128, refine_ctas=2),
                                dict(pipe_chunk=333, refine_ctas=4)],
                         ids=lambda kw: ",".join(f"{k}={v}" for k, v in kw.items()))
def test_same_results_as_plain_search(tiny, torch, kw):
    want = run(tiny, torch)
    got = run(tiny, torch, **kw)
    for a, b in zip(want, got):
        assert np.array_equal(a, b)


def test_on_a_side_stream_with_timing(tiny, torch):
    ix = tiny["ix"]
    want = run(tiny, torch)
    s = torch.cuda.Stream()
    ix.enable_timing(True)
    try:
        with torch.cuda.stream(s):
            got = run(tiny, torch, stream=s, pipe_chunk=200, refine_ctas=2)
        tm = ix.last_timing()
    finally:
        ix.enable_timing(False)
    for a, b in zip(want, got):
        assert np.array_equal(a, b)
    assert all(tm[k] > 0 for k in ("encode", "route", "select", "refine"))


def test_repeated_calls_reuse_buffers(tiny, torch):
    """Back-to-back pipelined calls on one stream: each sees its own inputs."""
    ix = tiny["ix"]
    dq = tiny["dq"]
    ix.set_params(**BASE)
    a = ix.search(dq[:500], 10, 64, 128)
    b = ix.search(dq[500:], 10, 64, 128)
    torch.cuda.synchronize()
    ix.set_params(**BASE, pipe_chunk=64)
    outs = [ix.search(dq[:500], 10, 64, 128), ix.search(dq[500:], 10, 64, 128),
            ix.search(dq[:500], 10, 64, 128)]
    torch.cuda.synchronize()
    ix.set_params()
    for (i0, d0), (i1, d1) in zip([a, b, a], outs):
        assert torch.equal(i0, i1) and torch.equal(d0, d1)


def test_argument_checks(tiny, torch):
    from paper_2608_15438_gb300 import neuroute as nr

    for bad in (dict(pipe_chunk=-1), dict(refine_ctas=-1), dict(refine_ctas=33)):
        with pytest.raises(nr.NRError):
            tiny["ix"].set_params(**bad)
    tiny["ix"].set_params()

"""nr_search_static: the search entry point that allocates nothing.

Some callers cannot allocate device memory while they serve queries (a host
framework or inference server owns the memory budget, or a latency-critical
loop cannot afford cudaMalloc / cudaFree, which may synchronise the device).
For them the library keeps its scratch in one fixed 32 MiB device array. This
test calls that entry point through the C ABI twice in a row and checks that
both calls return exactly what nr_search returns (ids and uint8 distances are
integers, so the comparison is exact), and that a request too large for the
array is refused before any work is enqueued.

The file name puts it last in collection order, so a run that stops at the
first failure has already run every other test; it also passes on its own in
a fresh process (it builds its own small index).
"""
import ctypes

import numpy as np
import pytest

import synth
from gpu_util import build_small, need_cuda

pytestmark = pytest.mark.gpu


def test_static_scratch_search_matches_workspace_search(tmp_path):
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, _ = build_small(tmp_path, "tiny", n=30000, bits=12, name="static")
    ix = nr.Index(path, 0)
    w = synth.WORKLOADS["tiny"]
    dq = torch.from_numpy(synth.queries(w, 300)).cuda()
    k, P, C = 10, 32, 64
    ref_ids, ref_d = ix.search(dq, k, P, C)
    ref_st = ix.query_stats(dq.shape[0])
    torch.cuda.synchronize()
    L = nr.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for _ in range(2):
        ids = torch.full((dq.shape[0], k), -7, dtype=torch.int64, device="cuda")
        d = torch.full((dq.shape[0], k), -7.0, dtype=torch.float32, device="cuda")
        st = L.nr_search_static(ix.h, ctypes.c_void_p(dq.data_ptr()), dq.shape[0], k, P, C,
                                ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(d.data_ptr()),
                                stream)
        assert st == nr.NR_OK
        torch.cuda.synchronize()
        assert torch.equal(ids, ref_ids)
        assert torch.equal(d, ref_d)
        assert torch.equal(ix.query_stats(dq.shape[0]), ref_st)
    assert ix.last_stats().nq == dq.shape[0]
    # a batch whose scratch would not fit in the fixed array is refused
    big = torch.zeros((20000, 128), dtype=torch.uint8, device="cuda")
    out_i = torch.empty((20000, k), dtype=torch.int64, device="cuda")
    out_d = torch.empty((20000, k), dtype=torch.float32, device="cuda")
    st = L.nr_search_static(ix.h, ctypes.c_void_p(big.data_ptr()), 20000, k, 1024, 1024,
                            ctypes.c_void_p(out_i.data_ptr()), ctypes.c_void_p(out_d.data_ptr()),
                            stream)
    assert st == -1  # NR_ERR_INVALID_ARG
    # the arguments are checked as nr_search checks them: the sequential
    # centroid stage refuses probe budgets above 2048 on both entry points
    ix.set_params(cent_mode=1)
    args = (ix.h, ctypes.c_void_p(dq.data_ptr()), 4, k, 3000, 64, ctypes.c_void_p(out_i.data_ptr()),
            ctypes.c_void_p(out_d.data_ptr()), stream)
    assert L.nr_search_static(*args) == -1
    assert L.nr_search(*args) == -1
    ix.close()


def test_static_scratch_search_global_sort_slabs(tmp_path):
    """Budgets whose candidate clusters exceed shared memory (P * K_max up to
    65,536, sorted in global slabs inside the fixed array) give nr_search's
    results too."""
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr

    path, _, _ = build_small(tmp_path, "tiny", n=30000, bits=12, k_max=16, t=4, name="slab")
    ix = nr.Index(path, 0)
    assert ix.k_max == 16
    w = synth.WORKLOADS["tiny"]
    dq = torch.from_numpy(synth.queries(w, 24)).cuda()
    k, P, C = 10, 4096, 256
    ref_ids, ref_d = ix.search(dq, k, P, C)
    ref_st = ix.query_stats(dq.shape[0])
    torch.cuda.synchronize()
    L = nr.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for _ in range(2):
        ids = torch.full((dq.shape[0], k), -7, dtype=torch.int64, device="cuda")
        d = torch.full((dq.shape[0], k), -7.0, dtype=torch.float32, device="cuda")
        st = L.nr_search_static(ix.h, ctypes.c_void_p(dq.data_ptr()), dq.shape[0], k, P, C,
                                ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(d.data_ptr()),
                                stream)
        assert st == nr.NR_OK
        torch.cuda.synchronize()
        assert torch.equal(ids, ref_ids) and torch.equal(d, ref_d)
        assert torch.equal(ix.query_stats(dq.shape[0]), ref_st)
    ix.close()


def test_static_scratch_search_multi_layer_encoder(tmp_path):
    """An index whose encoder has hidden layers after the first: the layer
    activations of its tensor-core encoder also live in the fixed array, and
    the results are nr_search's (fp32 distances by the same fmaf chain)."""
    torch = need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr
    from paper_2608_15438_gb300.builder import build_index, config
    from test_gpu_mlp import mlp_case

    base, q, weights, widths, b = mlp_case(512, (256, 128, 64), 12, 12_000)
    cfg = config("f32", base.shape[1], widths[0], b, 4, 16, mid=widths[1:])
    path = str(tmp_path / "mlp.nrix")
    build_index(cfg, base, weights, path)
    ix = nr.Index(path, 0)
    dq = torch.from_numpy(q).cuda()
    k, P, C = 10, 32, 64
    ref_ids, ref_d = ix.search(dq, k, P, C)
    torch.cuda.synchronize()
    L = nr.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for _ in range(2):
        ids = torch.full((dq.shape[0], k), -7, dtype=torch.int64, device="cuda")
        d = torch.full((dq.shape[0], k), -7.0, dtype=torch.float32, device="cuda")
        st = L.nr_search_static(ix.h, ctypes.c_void_p(dq.data_ptr()), dq.shape[0], k, P, C,
                                ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(d.data_ptr()),
                                stream)
        assert st == nr.NR_OK
        torch.cuda.synchronize()
        assert torch.equal(ids, ref_ids) and torch.equal(d, ref_d)
    ix.close()

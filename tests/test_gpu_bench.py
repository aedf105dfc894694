"""The benchmark's ground truth: exact k-NN over rows regenerated on the GPU
(group pre-selection, TF32 matmul for uint8) equals the oracle's brute force."""
import numpy as np
import pytest

import oracle
import synth
from gpu_util import need_cuda

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["tiny"])
def test_ground_truth_rows_is_exact(name):
    torch = need_cuda()
    import dataclasses

    import bench

    w = synth.WORKLOADS[name]
    w = dataclasses.replace(w, n=1 << 17)   # 128 groups of 1024 rows per chunk
    qs = synth.queries(w, 300)
    dq = torch.from_numpy(qs).cuda()
    got = bench.ground_truth_rows(torch, w, dq, 10, torch.device("cuda", 0), chunk=1 << 16)
    base = synth.base(w)
    ids_o, d_o = oracle.bruteforce(base, qs, 10)
    d_got = ((base[got].astype(np.int64) - qs[:, None, :].astype(np.int64)) ** 2).sum(-1)
    # same distances at every rank (ids may differ only among equal distances)
    assert np.array_equal(np.sort(d_got, 1), d_o.astype(np.int64))


def test_measurement_utilities_and_their_arguments():
    """The roofline denominators the benchmark measures in its run: a
    sequential read and random row gathers, each a plausible rate for one
    GPU (between 100 GB/s and 20 TB/s), gathers below the stream; arguments
    out of range are refused before any work."""
    need_cuda()
    from paper_2608_15438_gb300 import neuroute as nr

    read = nr.measure_read(0, 1 << 30, 2)
    gather = nr.measure_gather(0, 1 << 22, 96, n=4_000_000, reps=2)
    assert 100.0 < gather < read < 20_000.0
    for args in ((0, 1000, 2), (0, (1 << 20) + 8, 2), (0, 1 << 20, 0)):
        with pytest.raises(nr.NRError):
            nr.measure_read(*args)

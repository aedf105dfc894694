"""The GPU row generator (synth_cuda.cu) reproduces the host generator: uint8
rows exactly (also at row offsets near 1e9), fp32 rows to within one rounding
step (the GPU's and the host library's log/sin/cos may differ in the last bit
of a double)."""
import numpy as np
import pytest

import synth
from gpu_util import need_cuda

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,row0,n", [("u8-10m", 0, 200_000), ("u8-1b", 999_000_000, 5_000),
                                         ("u8-100m", 4_294_967_000, 1_000)])
def test_uint8_rows_equal_host(name, row0, n):
    torch = need_cuda()
    w = synth.WORKLOADS[name]
    dev = synth.DeviceRows(w, synth.SEED_DATA)
    got = dev.rows(row0, n).cpu().numpy()
    want = synth.mixture(w, synth.SEED_DATA, row0, n)
    assert np.array_equal(got, want)
    q = synth.DeviceRows(w, synth.SEED_QUERIES).rows(0, 1000).cpu().numpy()
    assert np.array_equal(q, synth.queries(w, 1000))


def test_fp32_rows_within_one_rounding_step():
    torch = need_cuda()
    w = synth.WORKLOADS["f32-10m"]
    got = synth.DeviceRows(w, synth.SEED_DATA).rows(123_456, 100_000).cpu().numpy()
    want = synth.mixture(w, synth.SEED_DATA, 123_456, 100_000)
    ulp = np.spacing(np.abs(want).astype(np.float32))
    assert np.all(np.abs(got - want) <= ulp)
    assert np.mean(got == want) > 0.999

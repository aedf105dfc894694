import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a)")


@pytest.fixture(scope="session", autouse=True)
def _native_built():
    import __graft_entry__

    __graft_entry__.build()


@pytest.fixture(scope="session")
def tiny_index(tmp_path_factory):
    """The 1e5 uint8 workload (b = 16) built once per session."""
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS["tiny"]
    base = synth.base(w)
    qs = synth.queries(w)
    W = synth.encoder_weights(w)
    path = str(tmp_path_factory.mktemp("idx") / "tiny.nrix")
    build_index(config(w.dtype, w.dim, w.hidden, w.bits, w.k_max, w.t), base, W, path)
    return {"path": path, "base": base, "queries": qs, "weights": W, "workload": w}

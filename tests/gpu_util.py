"""Helpers shared by the GPU tests (no method arithmetic here)."""
import os

import numpy as np
import pytest

import synth
from paper_2608_15438_gb300.builder import build_index, config


def need_cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def build_small(tmp_dir, workload="tiny", n=None, bits=None, k_max=None, t=None, name="idx"):
    """Build an index over the first n rows of a workload; returns (path, base)."""
    w = synth.WORKLOADS[workload]
    n = n or w.n
    base = synth.base(w, n)
    W1, b1, W2, b2 = synth.encoder_weights(w)
    b = bits or w.bits
    path = os.path.join(str(tmp_dir), f"{name}.nrix")
    info = build_index(config(w.dtype, w.dim, w.hidden, b, k_max or w.k_max, t or w.t), base,
                       (W1, b1, W2[:b], b2[:b]), path)
    return path, base, info


def recall(found, truth, k=10):
    r = []
    for f, g in zip(found, truth):
        g = set(int(v) for v in g[:k] if v >= 0)
        f = set(int(v) for v in f[:k] if v >= 0)
        r.append(len(f & g) / min(k, len(g)) if g else 1.0)
    return float(np.mean(r))


def cached_index(workload_name, tmp_root="/tmp"):
    """Full-size index of a workload, built once per machine and reused by
    content digest (workload definition + generator and builder sources)."""
    import hashlib

    from paper_2608_15438_gb300.builder import build_index, config

    w = synth.WORKLOADS[workload_name]
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    h = hashlib.sha256(repr(w).encode())
    for f in ("synth/synth.c", "paper_2608_15438_gb300/builder/nrbuild.cpp"):
        h.update(open(os.path.join(root, f), "rb").read())
    path = os.path.join(tmp_root, f"neuroute_{w.name}_{h.hexdigest()[:16]}.nrix")
    if not os.path.exists(path):
        base = synth.base(w)
        build_index(config(w.dtype, w.dim, w.hidden, w.bits, w.k_max, w.t, mid=w.mid), base,
                    synth.encoder_weights(w), path + f".tmp{os.getpid()}")
        os.replace(path + f".tmp{os.getpid()}", path)
    return path

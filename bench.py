"""Benchmark of the NeuRoute batched query path on GB300.

One step = one nr_search call over the workload's whole query batch (encode,
route, select, refine) with the index and the queries resident in HBM.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload u8-1b]
                  [--P 64 --C 128 --t-low 4] [--impl neuroute|reference] [--sweep]

Prints one JSON line (rank 0). Metric: queries per second at the workload's
Recall@10 ~ 0.90 operating point, plus the refinement kernel's achieved HBM
bandwidth against the measured copy bandwidth of this GPU.
Multi-GPU (torchrun): every rank is an independent replica with the full
index and its own query batch (weak scaling, no data-path collective).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "QPS at Recall@10~0.90 (batched query path); refine-scan HBM GB/s"

# operating points with Recall@10 in [0.88, 0.92], from `--sweep`, `--grid`
# and `--calibrate`: budgets P and C, early-stop t_low, and the centroid gate:
# m1 gives M(x) = m1 x; cq the calibrated curve at that quantile and cov the
# calibrated S_max at that coverage (Sec. 3.4), both fitted on CALIB_QUERIES
# held-out queries; neither: gate off
OPERATING_POINTS = {
    "tiny": dict(P=128, C=256, t_low=4),
    "u8-10m": dict(P=256, C=256, t_low=0, m1=4.0),
    "f32-10m": dict(P=512, C=256, t_low=16),
    "u8-100m": dict(P=1024, C=256, t_low=32),
    "u8-1b": dict(P=1024, C=1024, t_low=80, cq=0.9, cov=0.99),
    "u8-30m": dict(P=1024, C=1024, t_low=80, cq=0.9, cov=0.99),  # profiling proxy of u8-1b
    # the random four-hidden-layer encoder in 1536 dims is a weak hash: the band
    # needs P = 2048 (0.876 at most with P = 1024)
    "f32-1536": dict(P=2048, C=2048, t_low=256),
    "f32-1536-1m": dict(P=2048, C=2048, t_low=256),  # profiling proxy of f32-1536
}
DEFAULT_POINT = dict(P=64, C=128, t_low=4)
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal
CALIB_QUERIES = 10000
CALIB_BINS = 16


EXEC_KEYS = ("pipe_chunk", "refine_ctas")  # nr_params fields that change no result

# encoder weights of the run: the workload's seeded weights, or a trained
# encoder's (--weights, written by paper_2608_15438_gb300.train)
ENCODER = {"weights": None, "source": "seeded N(0, 1/fan_in)"}


def workload_weights(w):
    """The encoder weights the run indexes and queries with."""
    import synth

    return ENCODER["weights"] if ENCODER["weights"] is not None else synth.encoder_weights(w)


def method_kw(kw):
    """The parameters of the method itself (the oracle's), without the
    library's execution settings."""
    return {k: v for k, v in kw.items() if k not in EXEC_KEYS}


def op_params(w, ix=None, t_low=None, calib=None, k=10):
    """nr_params keyword arguments of the workload's operating point. A
    calibrated point fits its curve and cutoff on the GPU index ix (or on
    given observations), outside any timed region."""
    op = OPERATING_POINTS.get(w.name, DEFAULT_POINT)
    kw = {"t_low": op["t_low"] if t_low is None else t_low}
    if op.get("m1") is not None:
        kw.update(gate_m0=0.0, gate_m1=op["m1"])
    if op.get("cq") is not None or op.get("cov") is not None:
        if calib is None:
            if ix is None:
                raise SystemExit(f"{w.name}: the calibrated operating point needs the GPU index")
            calib = calibration_observations(w, ix, op["P"], op["C"], k)
        kw.update(calibrated_params(calib, op.get("cq"), op.get("cov"), CALIB_BINS))
    return kw


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="u8-1b")
    ap.add_argument("--P", type=int, default=None)
    ap.add_argument("--C", type=int, default=None)
    ap.add_argument("--t-low", type=int, default=None)
    ap.add_argument("--k", type=int, default=10)
    ap.add_argument("--nq", type=int, default=None)
    ap.add_argument("--impl", default="neuroute", choices=["neuroute", "reference"])
    ap.add_argument("--sweep", action="store_true")
    ap.add_argument("--sweep-gate", action="store_true",
                    help="sweep the centroid gate M(x) = m1 x around the (P, C) grid")
    ap.add_argument("--grid", default=None,
                    help="sweep grid 'P=..;C=..;t_low=..;m1=..' (comma lists, m1 'none' = gate off)")
    ap.add_argument("--index", default=None, help="reuse an index file (host builder)")
    ap.add_argument("--builder", default="gpu", choices=["gpu", "host"],
                    help="build the index on the GPU from generated rows (default) or on the host")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-gt", action="store_true", help="skip ground truth (profiling runs)")
    ap.add_argument("--encode", type=int, default=0,
                    help="time only the tensor-core encoder over this many base vectors")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--weights", default=None,
                    help="encoder weights (.npz from paper_2608_15438_gb300.train) instead of the "
                         "workload's seeded ones")
    ap.add_argument("--calibrate", type=int, default=0,
                    help="calibrate M(x) and S_max on this many held-out queries (Sec. 3.4; "
                         "default 10,000 when the operating point is calibrated); grid keys "
                         "cq=<quantile> and cov=<coverage> select the fitted curve and cutoff")
    ap.add_argument("--calib-budget", default=None, help="'P,C' of the high-recall target run")
    ap.add_argument("--calib-bins", type=int, default=CALIB_BINS)
    ap.add_argument("--cq", type=float, default=None,
                    help="timed run: calibrated gate at this quantile (needs --calibrate)")
    ap.add_argument("--cov", type=float, default=None,
                    help="timed run: calibrated S_max at this coverage (needs --calibrate)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(x, world, device=None):
    """The largest of the ranks' values of x (every rank calls it; x itself
    at world size 1): the job's time is its slowest rank's."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank, world, seconds):
    """Whole-job throughput: the units every rank processed over the job's time."""
    return units_per_rank * world / seconds


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() in ("active", "1", "yes"):
                        reasons.add(n)
            os.remove(self.path)
        except Exception:
            pass
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def index_path(w):
    """Index file named by a digest of everything that determines its bytes."""
    h = hashlib.sha256(repr(w).encode())
    for f in ("synth/synth.c", "paper_2608_15438_gb300/builder/nrbuild.cpp"):
        h.update(open(os.path.join(ROOT, f), "rb").read())
    if ENCODER["weights"] is not None:
        for a in ENCODER["weights"][:4]:
            h.update(np.ascontiguousarray(a).tobytes())
    return os.path.join(tempfile.gettempdir(), f"neuroute_{w.name}_{h.hexdigest()[:16]}.nrix")


def build_or_load_index(w, path, rank, world):
    import synth
    from paper_2608_15438_gb300.builder import build_index, config

    if rank == 0 and not os.path.exists(path):
        base = synth.base(w)
        info = build_index(config(w.dtype, w.dim, w.hidden, w.bits, w.k_max, w.t, mid=w.mid), base,
                           workload_weights(w), path + ".tmp")
        os.replace(path + ".tmp", path)
        del base
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    return path


def gpu_index(w, torch, nr, dev):
    """The workload's index built on the GPU (neuroute_build.h) from rows that
    the GPU generator draws twice: once to encode, once to store."""
    import synth
    from paper_2608_15438_gb300.builder import config

    d = dev.index or 0
    gen = synth.DeviceRows(w, synth.SEED_DATA, device=d)
    bd = nr.Builder(config(w.dtype, w.dim, w.hidden, w.bits, w.k_max, w.t, mid=w.mid), w.n,
                    workload_weights(w), d)
    chunk = min(w.n, (4 << 30) // w.row_bytes)
    buf = torch.empty((chunk, w.dim), dtype=torch.uint8 if w.dtype == "u8" else torch.float32,
                      device=dev)
    for r0 in range(0, w.n, chunk):
        m = min(chunk, w.n - r0)
        bd.encode(gen.rows(r0, m, out=buf), r0)
    torch.cuda.synchronize()
    info = bd.finish()
    for r0 in range(0, w.n, chunk):
        m = min(chunk, w.n - r0)
        bd.place(gen.rows(r0, m, out=buf), r0)
    ix = bd.end()
    del buf
    torch.cuda.empty_cache()
    return ix, info


def ground_truth_rows(torch, w, dq, k, dev, chunk=1 << 22, qblock=2500, group=1024):
    """Exact k-NN of the queries over the whole base, rows regenerated on the
    GPU chunk by chunk. Distances are |x|^2 - 2 q.x (the query norm does not
    change the order); for uint8 rows every product and partial sum is an
    integer below 2^24, so the TF32 tensor-core matmul is exact. Per chunk the
    k nearest rows lie in the k groups of `group` rows with the smallest
    minimum distance, so the top-k runs only over those groups."""
    import synth

    gen = synth.DeviceRows(w, synth.SEED_DATA, device=dev.index or 0)
    # at most about 512 MB of rows a chunk, in whole groups
    chunk = max(group * 16, min(chunk, ((512 << 20) // w.row_bytes) // group * group))
    Q = dq.float()
    nq = Q.shape[0]
    best_d = torch.full((nq, k), float("inf"), device=dev)
    best_i = torch.full((nq, k), -1, dtype=torch.int64, device=dev)
    tf32 = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = w.dtype == "u8"
    try:
        for r0 in range(0, w.n, chunk):
            m = min(chunk, w.n - r0)
            X = gen.rows(r0, m).float()
            bn = (X * X).sum(1)
            for q0 in range(0, nq, qblock):
                q1 = min(nq, q0 + qblock)
                dmat = bn[None, :] - 2.0 * (Q[q0:q1] @ X.T)
                if m % group == 0 and m // group > k:
                    g = dmat.view(q1 - q0, m // group, group)
                    top_g = torch.topk(g.amin(2), k, dim=1, largest=False).indices
                    cand = torch.gather(g, 1, top_g[:, :, None].expand(-1, -1, group))
                    v, i = torch.topk(cand.reshape(q1 - q0, -1), k, dim=1, largest=False)
                    i = torch.gather(top_g, 1, i // group) * group + i % group
                else:
                    v, i = torch.topk(dmat, min(k, m), dim=1, largest=False)
                cv = torch.cat([best_d[q0:q1], v], 1)
                ci = torch.cat([best_i[q0:q1], i + r0], 1)
                vv, ii = torch.topk(cv, k, dim=1, largest=False)
                best_d[q0:q1] = vv
                best_i[q0:q1] = torch.gather(ci, 1, ii)
                del dmat
            del X
        torch.cuda.synchronize()
    finally:
        torch.backends.cuda.matmul.allow_tf32 = tf32
    return best_i.cpu().numpy()


def oracle_subindex(w, ix, qs, P, kw, path):
    """Sub-index of the buckets that the oracle probes for queries qs: the
    oracle's own logits (double-precision encoder) and probe lists pick the
    codes, the library copies those buckets out (nr_index_extract). The oracle
    then answers these queries on the file exactly as on the whole index."""
    import oracle
    import synth

    lg = oracle.encode_weights(workload_weights(w), w.in_scale, qs)
    tau = ix.thresholds()
    p = oracle.params(**method_kw(kw))
    codes = np.concatenate([oracle.probe_list(lg[i], tau, P, p)[0] for i in range(len(qs))])
    rows, _ = ix.extract(codes, path)
    return lg, rows


def ground_truth(torch, base_t, q_t, k, dtype):
    """Exact k-NN by brute force on the GPU (torch fp32 matmul; exact for uint8
    data, whose dot products and norms are integers below 2^24)."""
    nb = base_t.shape[0]
    bf = base_t.float()
    bn = (bf * bf).sum(1)
    out = []
    step = max(1, int(2e9 // max(nb, 1)))
    for i in range(0, q_t.shape[0], step):
        qf = q_t[i:i + step].float()
        d = (qf * qf).sum(1, keepdim=True) + bn[None, :] - 2.0 * (qf @ bf.T)
        out.append(torch.topk(d, k, dim=1, largest=False).indices.cpu())
        del d
    return torch.cat(out).numpy()


def recall_at(found, truth, k=10):
    """Recall@k (Sec. 4.4): |R & G| / min(k, |G|) over the unique valid ids of
    the first k found (R) and true (G) neighbours, averaged over queries."""
    r = []
    for f, g in zip(found, truth):
        g = set(int(v) for v in g[:k] if v >= 0)
        f = set(int(v) for v in f[:k] if v >= 0)
        r.append(len(f & g) / min(k, len(g)) if g else 1.0)
    return float(np.mean(r))


def refine_sources_digest():
    """sha256 over the sources that define the refine kernel."""
    h = hashlib.sha256()
    for f in ("nr_refine.cu", "nrq_refine.cuh", "nrq_common.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2608_15438_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def traffic_from_profile(workload, P, C, algorithmic_bytes, launches=1):
    """Per-launch DRAM bytes of the refine kernel and where they come from:
    a committed ncu capture of this workload's operating point (valid only
    while the kernel source is unchanged since the capture and the capture
    scanned the same candidates), else a capture of a smaller proxy on the
    same sources scaled by the candidate bytes (the scan reads each
    candidate row once, so its traffic grows with them); (None, None)
    without either."""
    path = os.path.join(ROOT, "profiles", "refine_traffic.json")
    try:
        rec = json.load(open(path))
        caps = rec.get("captures", {})
        digest = refine_sources_digest()
        e = caps.get(f"{workload}/P{P}/C{C}")
        if (e is not None and e.get("sources_sha256") == digest and e.get("launches", 1) == launches
                and e.get("algorithmic_bytes_per_launch") * launches == algorithmic_bytes):
            return e.get("bytes_per_launch"), "ncu capture of this workload"
        for key, e in caps.items():
            if e.get("sources_sha256") == digest and e.get("scales_to", {}).get(workload):
                ratio = e["bytes_per_launch"] / e["algorithmic_bytes_per_launch"]
                return (ratio * algorithmic_bytes / launches,
                        f"ncu capture of {key} scaled by candidate bytes (DRAM / algorithmic "
                        f"{ratio:.3f} there)")
        return None, None
    except Exception:
        return None, None


def cpu_baseline(w, path, queries, k, P, C, kw, seconds, truth=None):
    import oracle

    orc = oracle.Index(path)
    t_low = kw.get("t_low")
    p = oracle.params(**method_kw(kw))
    cores = os.cpu_count() or 1
    n = 16
    t = time.perf_counter()
    orc.search(queries[:n], k, P, C, p, nthreads=cores)
    dt = max(time.perf_counter() - t, 1e-6)
    n2 = int(min(len(queries), max(n, n * seconds / dt)))
    t = time.perf_counter()
    ids, _, _ = orc.search(queries[:n2], k, P, C, p, nthreads=cores)
    dt2 = time.perf_counter() - t
    v1, n1, dt1 = one_thread_rate(orc, queries, n2, dt2, cores, k, P, C, p, seconds)
    res = {"value": n2 / dt2, "unit": "queries/s", "cores": cores, "kind": "oracle",
           "value_1_thread": v1,
           "sample": f"first {n2} of {len(queries)} queries of {w.name}, P={P} C={C} t_low={t_low}, "
                     f"{cores} threads, {dt2:.1f} s; one thread: first {n1}, {dt1:.1f} s"}
    orc.close()
    return res, ids


def one_thread_rate(orc, queries, n, dt, cores, k, P, C, p, seconds):
    """The oracle's rate on one thread over a prefix of the timed sample sized
    to about a quarter of `seconds` (from the all-core rate at perfect scaling)."""
    per_q = dt * cores / max(n, 1)
    n1 = int(min(n, max(2, 0.25 * seconds / max(per_q, 1e-9))))
    t = time.perf_counter()
    orc.search(queries[:n1], k, P, C, p, nthreads=1)
    dt1 = max(time.perf_counter() - t, 1e-9)
    return n1 / dt1, n1, dt1


def calibrate_subindex(w, ix, queries, k, P, C, kw, seconds, path, row_budget):
    """Number of queries whose oracle run takes about `seconds` on the host
    cores, bounded by the query count and by a sub-index of at most
    row_budget rows (estimated from the first 16 queries)."""
    import oracle

    n = min(16, len(queries))
    lg, rows = oracle_subindex(w, ix, queries[:n], P, kw, path)
    orc = oracle.Index(path)
    t = time.perf_counter()
    orc.search(queries[:n], k, P, C, oracle.params(**method_kw(kw)), logits=lg, nthreads=os.cpu_count() or 1)
    dt = max(time.perf_counter() - t, 1e-6)
    orc.close()
    per_q = max(1.0, rows / n)
    return int(min(len(queries), max(n, row_budget / per_q), max(n, n * seconds / dt)))


def cpu_baseline_subindex(w, ix, queries, k, P, C, kw, seconds, row_budget=100_000_000):
    """The oracle timed on the host cores for a bounded query sample, on the
    sub-index of the buckets those queries probe (the index may be too large
    for host memory), with the timed run's parameters kw."""
    import oracle

    t_low = kw.get("t_low")
    p = oracle.params(**method_kw(kw))
    cores = os.cpu_count() or 1
    with tempfile.TemporaryDirectory() as td:
        sub = os.path.join(td, "sub.nrix")
        n2 = calibrate_subindex(w, ix, queries, k, P, C, kw, seconds, sub, row_budget)
        _, rows = oracle_subindex(w, ix, queries[:n2], P, kw, sub)
        orc = oracle.Index(sub)
        t = time.perf_counter()
        orc.search(queries[:n2], k, P, C, p, nthreads=cores)
        dt1 = max(time.perf_counter() - t, 1e-6)
        # repeat the sample (when the sub-index bound limits it) to about `seconds`
        reps = int(max(1, min(50, seconds / dt1)))
        t = time.perf_counter()
        for _ in range(reps):
            orc.search(queries[:n2], k, P, C, p, nthreads=cores)
        dt2 = time.perf_counter() - t
        v1, n1, dt1 = one_thread_rate(orc, queries, n2, dt2 / reps, cores, k, P, C, p, seconds)
        orc.close()
    return {"value": n2 * reps / dt2, "unit": "queries/s", "cores": cores, "kind": "oracle",
            "value_1_thread": v1,
            "sample": f"first {n2} of {len(queries)} queries of {w.name} (oracle encoder included), "
                      f"{reps} passes, P={P} C={C} t_low={t_low}, {cores} threads, {dt2:.1f} s, on "
                      f"the {rows}-row sub-index of the buckets they probe; one thread: first {n1}, "
                      f"{dt1:.1f} s"}


def run_reference(args, w, rank, world):
    """The oracle timed on the host cores (the CPU reference arm)."""
    if rank != 0:
        return 0
    import synth

    P, C, t_low = op_point(args, w)
    nq = args.nq or w.nq
    nq_all = nq
    qs = synth.queries(w, nq)
    import oracle

    tmpdir = None
    if args.builder == "gpu" and not args.index:
        # the index is built on the GPU (setup, outside the timed region); the
        # oracle answers a bounded query sample from the sub-index of the
        # buckets those queries probe
        import torch

        import __graft_entry__

        __graft_entry__.build()
        from paper_2608_15438_gb300 import neuroute as nr

        dev = torch.device("cuda", 0)
        gix, _ = gpu_index(w, torch, nr, dev)
        kw0 = op_params(w, gix, t_low, k=args.k)
        tmpdir = tempfile.TemporaryDirectory()
        path = os.path.join(tmpdir.name, "sub.nrix")
        per_step = max(8.0, 120.0 / max(1, args.steps + args.warmup))
        nsub = calibrate_subindex(w, gix, qs, args.k, P, C, kw0, per_step, path, 100_000_000)
        oracle_subindex(w, gix, qs[:nsub], P, kw0, path)
        gix.close()
        del gix
        torch.cuda.empty_cache()
        qs = qs[:nsub]
        nq = nsub
    else:
        path = args.index or index_path(w)
        build_or_load_index(w, path, 0, 1)
    orc = oracle.Index(path)
    note = ("; sub-index of the buckets these queries probe, index built on the GPU"
            if tmpdir is not None else "")
    kw = kw0 if tmpdir is not None else op_params(w, t_low=t_low)
    p = oracle.params(**method_kw(kw))
    cores = os.cpu_count() or 1
    n = 16
    t = time.perf_counter()
    orc.search(qs[:n], args.k, P, C, p, nthreads=cores)
    dt = max(time.perf_counter() - t, 1e-6)
    per_step = max(8.0, 120.0 / max(1, args.steps + args.warmup))
    ns = int(min(nq, max(n, n * per_step / dt)))
    for _ in range(args.warmup):
        orc.search(qs[:ns], args.k, P, C, p, nthreads=cores)
    times = []
    for _ in range(args.steps):
        t = time.perf_counter()
        orc.search(qs[:ns], args.k, P, C, p, nthreads=cores)
        times.append(time.perf_counter() - t)
    tot = sum(times)
    v = ns * args.steps / tot
    line = {"impl": "reference", "metric": METRIC, "value": v,
            "unit": "queries/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u8" if w.dtype == "u8" else "f32", "data": "synthetic",
            "config": {"workload": w.name, "nq_per_step": ns, "P": P, "C": C, "t_low": t_low, "k": args.k,
                       "gate_m1": kw.get("gate_m1"), "gate_curve": kw.get("gate_curve"),
                       "s_max": kw.get("s_max")},
            "cpu_baseline": {"value": v, "unit": "queries/s", "cores": cores, "kind": "oracle",
                             "sample": f"first {ns} of {nq_all} queries per step{note}"},
            "e2e": {"value": v, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    orc.close()
    if tmpdir is not None:
        tmpdir.cleanup()
    return 0


def encode_bench(args, w, torch, nr, dev):
    """Throughput of the encoder (K1, tensor cores) over a batch of base
    vectors, the operation an index build runs over the whole base."""
    import dataclasses

    import synth

    # the encoder does not depend on the index contents: a small index over
    # the workload's first rows carries the same weights
    ix, _ = gpu_index(dataclasses.replace(w, n=min(w.n, 100_000)), torch, nr, dev)
    x = synth.DeviceRows(w, synth.SEED_DATA, device=dev.index or 0).rows(0, args.encode)
    out = torch.empty((args.encode, w.bits), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    L = nr.lib()
    import ctypes

    def run():
        st = L.nr_encode(ix.h, ctypes.c_void_p(x.data_ptr()), args.encode, ctypes.c_void_p(out.data_ptr()),
                         ctypes.c_void_p(stream.cuda_stream))
        if st != 0:
            raise RuntimeError(f"nr_encode failed {st}")

    for _ in range(max(3, args.warmup)):
        run()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(stream)
    for _ in range(args.steps):
        run()
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    dims = [w.dim, w.hidden, *getattr(w, "mid", ()), w.bits]
    flops = 2.0 * args.encode * sum(a * c for a, c in zip(dims[:-1], dims[1:]))
    peaks, src = measured_peaks()
    tf = flops / (ms / 1e3) / 1e12
    print(json.dumps({"metric": "encoder TFLOP/s (fp16 tensor cores, fp32 accumulate)", "value": tf,
                      "unit": "TFLOP/s", "rows": args.encode, "ms_per_launch": ms,
                      "roofline": {"bound": "tensor", "achieved": tf, "peak": peaks.get("bf16_tflops"),
                                   "unit": "TFLOP/s", "frac": tf / peaks.get("bf16_tflops"),
                                   "peak_source": src + " bf16 dense (fp16 dense runs at the same nominal rate)"},
                      "config": {"workload": w.name, "layers": dims}}), flush=True)
    return 0


def calibration_observations(w, ix, P, C, k, nq=CALIB_QUERIES, budget=None, bins=CALIB_BINS):
    """Observations for the calibrated gate and cutoff (Sec. 3.4) from nq
    held-out calibration queries, targets from a high-recall run of the search
    (budgets 2P and 4C by default, gate and early stop off)."""
    import torch

    import synth
    from paper_2608_15438_gb300 import calibrate as cal

    t0 = time.time()
    dev = torch.device("cuda", ix.device)
    cq = torch.from_numpy(synth.calib_queries(w, nq)).to(dev)
    # the target run's probe budget: twice the operating point's, with at most
    # 16,384 candidate clusters a query, which bounds the calibration's cost
    cP, cC = budget or (min(4096, 2 * P, 16384 // ix.k_max), min(4096, 4 * C))
    lg = ix.encode(cq)
    targets = cal.targets_high_recall(ix, cq, lg, k, cP, cC)
    scores, x, y = cal.observations(ix, lg, targets)
    torch.cuda.synchronize()
    summary = {"nq": nq, "budget": [cP, cC], "seconds": round(time.time() - t0, 2),
               "n_gated": int((~np.isnan(x)).sum()),
               "curves": {q: cal.fit_gate(x, y, bins, q) for q in (0.9, 0.95, 0.99)},
               "s_max": {c: [float(v) for v in cal.fit_s_max(scores, c)] for c in (0.95, 0.99, 0.999)}}
    print(json.dumps({"calibration": summary}), file=sys.stderr, flush=True)
    return {"scores": scores, "x": x, "y": y, "nq": nq, "budget": [cP, cC]}


def calibrated_params(calib, cq, cov, bins=CALIB_BINS):
    """nr_params keywords of the calibrated gate (quantile cq) and cutoff
    (coverage cov); either may be None."""
    from paper_2608_15438_gb300 import calibrate as cal

    kw = {}
    if cq is None and cov is None:
        return kw
    if calib is None:
        raise SystemExit("cq/cov need calibration observations (--calibrate)")
    if cq is not None:
        curve = cal.fit_gate(calib["x"], calib["y"], bins, cq)
        if curve is not None:
            kw["gate_curve"] = curve
    if cov is not None:
        s_max = cal.fit_s_max(calib["scores"], cov)[0]
        if s_max is not None:
            kw["s_max"] = float(s_max)
    return kw


def op_point(args, w):
    op = OPERATING_POINTS.get(w.name, DEFAULT_POINT)
    return (args.P or op["P"], args.C or op["C"], op["t_low"] if args.t_low is None else args.t_low)


def main():
    args = parse()
    import synth

    w = synth.WORKLOADS[args.workload]
    if args.weights:
        from paper_2608_15438_gb300 import train

        ENCODER["weights"] = train.load_weights(args.weights)
        ENCODER["source"] = f"trained with L_sim ({os.path.basename(args.weights)})"
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("gloo" if args.impl == "reference" else "nccl")
    if args.impl == "reference":
        rc = run_reference(args, w, rank, world)
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()
        return rc

    import torch

    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_15438_gb300 import neuroute as nr

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if args.encode:
        return encode_bench(args, w, torch, nr, dev)
    P, C, t_low = op_point(args, w)
    k = args.k
    gpu_built = args.builder == "gpu" and not args.index
    t0 = time.time()
    if gpu_built:
        path = None
        ix, build_info = gpu_index(w, torch, nr, dev)
    else:
        path = args.index or index_path(w)
        build_or_load_index(w, path, rank, world)
        ix = nr.Index(path, local)
        build_info = None
    t_build = time.time() - t0
    nq = args.nq or w.nq
    # each rank searches its own batch of the query distribution
    qs = synth.mixture(w, synth.SEED_QUERIES, rank * nq, nq)
    dq = torch.from_numpy(qs).to(dev)
    ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    dd = torch.empty((nq, k), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    # ground truth (outside any timed region)
    truth = None
    t0 = time.time()
    if not args.no_gt:
        if gpu_built:
            truth = ground_truth_rows(torch, w, dq, k, dev)
        else:
            base_np = synth.base(w)
            base_t = torch.from_numpy(base_np).to(dev)
            del base_np
            truth = ground_truth(torch, base_t, dq, k, w.dtype)
            del base_t
        torch.cuda.empty_cache()
    t_gt = time.time() - t0
    print(json.dumps({"setup_s": {"index_build": round(t_build, 2), "ground_truth": round(t_gt, 2)},
                      "index": build_info, "n_clusters": ix.n_clusters}), file=sys.stderr, flush=True)

    op = OPERATING_POINTS.get(w.name, DEFAULT_POINT)
    calibrated_op = op.get("cq") is not None or op.get("cov") is not None
    calib = None
    if args.calibrate or calibrated_op or args.cq is not None or args.cov is not None:
        budget = tuple(int(v) for v in args.calib_budget.split(",")) if args.calib_budget else None
        calib = calibration_observations(w, ix, P, C, k, nq=args.calibrate or CALIB_QUERIES,
                                         budget=budget, bins=args.calib_bins)

    if args.sweep or args.sweep_gate or args.grid:
        import itertools

        def num(v):
            return None if v == "none" else (float(v) if ("." in v or "e" in v or v == "inf") else int(v))

        if args.grid:
            # "P=..;C=..;t_low=..;m1=..;<any nr_params field>=.." (comma lists)
            g = {k: [num(v) for v in vals.split(",")]
                 for k, vals in (part.split("=") for part in args.grid.split(";"))}
        elif args.sweep_gate:
            g = {"P": [128, 256, 512], "C": [128, 256, 1024], "t_low": [0, 32, 64],
                 "m1": [None, 0.5, 1.0, 2.0, 4.0]}
        else:
            g = {"P": [64, 128, 256, 512, 1024] if w.bits <= 20 else [256, 512, 1024],
                 "C": [256, 512, 1024, 2048] if w.bits <= 20 else [256, 1024],
                 "t_low": [0, 8, 16, 32, 64], "m1": [None]}
            if w.k_max == 1:  # no bucket-local clustering: C never binds
                g["P"], g["C"] = [64, 128, 256, 512, 1024, 2048], [256]
        g.setdefault("P", [P])
        g.setdefault("C", [C])
        g.setdefault("m1", [None])
        names = list(g)
        for combo in itertools.product(*(g[k] for k in names)):
            cfg = dict(zip(names, combo))
            Pp, Cc, m1 = cfg["P"], cfg["C"], cfg["m1"]
            if Pp * ix.k_max > 65536:
                continue
            kw = {k: v for k, v in cfg.items() if k not in ("P", "C", "m1", "cq", "cov")}
            if m1 is not None:
                kw.update(gate_m0=0.0, gate_m1=m1)
            kw.update(calibrated_params(calib, cfg.get("cq"), cfg.get("cov"), args.calib_bins))
            try:
                ix.set_params(**kw)
                ix.search(dq, k, Pp, Cc, out=(ids, dd))
            except nr.NRError as ex:
                print(json.dumps({**cfg, "error": str(ex)}), flush=True)
                continue
            torch.cuda.synchronize()
            els = []
            for _ in range(3):  # median of three
                t = time.perf_counter()
                ix.search(dq, k, Pp, Cc, out=(ids, dd))
                torch.cuda.synchronize()
                els.append(time.perf_counter() - t)
            el = statistics.median(els)
            st = ix.last_stats()
            print(json.dumps({**cfg, "recall": recall_at(ids.cpu().numpy(), truth, k), "qps": nq / el,
                              "cand_per_q": st.candidates / nq, "clusters_per_q": st.clusters / nq}),
                  flush=True)
        return 0

    if args.cq is not None or args.cov is not None:
        cq, cov, bins = args.cq, args.cov, args.calib_bins
        kw = {"t_low": t_low, **calibrated_params(calib, cq, cov, bins)}
    else:
        cq, cov, bins = op.get("cq"), op.get("cov"), CALIB_BINS
        kw = op_params(w, ix, t_low, calib=calib, k=k)
    ix.set_params(**kw)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(max(3, args.warmup)):
        ix.search(dq, k, P, C, out=(ids, dd), stream=stream)
    torch.cuda.synchronize()
    rec = None if truth is None else recall_at(ids.cpu().numpy(), truth, k)
    st = ix.last_stats()
    ix.enable_timing(True)
    launches0 = ix.kernel_launches()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    refine_ms = []
    stage_ms = {"encode": 0.0, "route": 0.0, "select": 0.0, "refine": 0.0}
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(torch.cuda.current_device() if "CUDA_VISIBLE_DEVICES" not in os.environ else local) as clk:
        for i in range(args.steps):
            flush.random_(0, 255)  # evict L2 (129 MB) between timed steps
            ev[i][0].record(stream)
            ix.search(dq, k, P, C, out=(ids, dd), stream=stream)
            ev[i][1].record(stream)
            tm = ix.last_timing()
            refine_ms.append(tm["refine"])
            for kk in stage_ms:
                stage_ms[kk] += tm[kk]
        torch.cuda.synchronize()
    launches = ix.kernel_launches() - launches0
    step_ms = [a.elapsed_time(b) for a, b in ev]
    tot_ms = sum(step_ms)
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    tot_ms = max_over_ranks(tot_ms, world, dev)
    value = job_rate(nq * args.steps, world, tot_ms / 1e3)

    # end to end through the host-buffer entry point (copies inside the timed region)
    hq = torch.from_numpy(qs).pin_memory()
    hid = torch.empty((nq, k), dtype=torch.int64).pin_memory()
    hd = torch.empty((nq, k), dtype=torch.float32).pin_memory()
    ix.search_host(hq, k, P, C, out=(hid, hd))
    e2e_t = []
    for _ in range(args.steps):
        flush.random_(0, 255)
        torch.cuda.synchronize()
        t = time.perf_counter()
        ix.search_host(hq, k, P, C, out=(hid, hd))
        e2e_t.append(time.perf_counter() - t)
    e2e_v = job_rate(nq * args.steps, world, max_over_ranks(sum(e2e_t), world, dev))

    cand = st.candidates
    row_bytes = w.row_bytes
    # refinement launches per step: one per pipelined chunk
    pc = kw.get("pipe_chunk", 0) or 0
    n_ref = -(-nq // pc) if 0 < pc < nq else 1
    refine_avg_ms = sum(refine_ms) / len(refine_ms) / n_ref
    achieved = cand * row_bytes / n_ref / (refine_avg_ms / 1e3) / 1e9
    peaks, peak_src = measured_peaks()
    traffic, traffic_src = traffic_from_profile(w.name, P, C, cand * row_bytes, n_ref)
    # select per launch: centroid rows of every scored cluster and the
    # directory pair of every probe
    sel_bytes = (st.scored * w.bits * 4 + st.probes * 8) / n_ref
    sel_avg_ms = stage_ms["select"] / args.steps / n_ref
    sel_gbs = sel_bytes / (sel_avg_ms / 1e3) / 1e9 if sel_avg_ms > 0 else None
    # the random-row read rate of this GPU over an array of the centroids' shape
    # (rows of 4b bytes rounded up to 16, the granule of the measurement)
    gather_gbs = nr.measure_gather(local, max(1 << 20, ix.n_clusters), (w.bits * 4 + 15) // 16 * 16)
    # the sequential-read rate of this GPU (8 GiB, L2 flushed): the scan's
    # bytes are reads of long runs
    read_gbs = nr.measure_read(local)
    out = {
        "metric": METRIC,
        "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": tot_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "u8" if w.dtype == "u8" else "f32", "data": "synthetic",
        "config": {"workload": w.name, "N": w.n, "D": w.dim, "nq": nq, "k": k, "bits": w.bits,
                   "hidden": w.hidden, "K_max": w.k_max, "encoder": ENCODER["source"],
                   "P": P, "C": C, "t_low": t_low,
                   "gate_m1": kw.get("gate_m1"), "gate_curve": kw.get("gate_curve"),
                   "s_max": kw.get("s_max"),
                   "calibration": (None if cq is None and cov is None else
                                   {"queries": calib["nq"], "target_budget": calib["budget"],
                                    "quantile": cq, "coverage": cov, "bins": bins,
                                    "held_out": "synthetic query stream of its own seed"}),
                   "round": 256, "recall_at_10": rec, "cand_per_query": cand / nq,
                   "l2": "flushed between timed steps (256 MB write)",
                   "parallelism": f"replicas x{world} (queries sharded, no collective)"},
        "roofline": {"kernel": "nr_refine", "bound": "hbm", "achieved": achieved,
                     "peak": peaks.get("hbm_gbs"), "unit": "GB/s",
                     "frac": achieved / peaks.get("hbm_gbs"),
                     "peak_source": f"{peak_src} hbm_gbs (a device copy's read + write bytes per "
                                    "second); the scan reads, so it can exceed it",
                     "frac_of_nominal": achieved / NOMINAL_HBM_GBS,
                     "stream_read_gbs": read_gbs, "frac_of_stream_read": achieved / read_gbs,
                     "stream_read_source": "measured in this run: an 8 GiB sequential read, L2 "
                                           "flushed, best of 5 (nr_measure_read)",
                     "traffic": traffic, "traffic_source": traffic_src,
                     "algorithmic_bytes_per_launch": cand * row_bytes / n_ref,
                     "avg_launch_ms": refine_avg_ms, "launches_per_step": n_ref},
        # the centroid stage's own roofline (Sec. 3.5's C_q b floats a query
        # plus one directory pair per probe), against the random-row read
        # rate of this GPU (its bytes are random row gathers) and, for
        # scale, against the copy bandwidth
        "roofline_select": {"kernel": "nr_select", "bound": "hbm random gather",
                            "achieved": sel_gbs, "peak": gather_gbs, "unit": "GB/s",
                            "frac": (sel_gbs / gather_gbs if sel_gbs and gather_gbs else None),
                            "frac_of_copy": (sel_gbs / peaks.get("hbm_gbs") if sel_gbs else None),
                            "peak_source": f"measured in this run: random "
                                           f"{(w.bits * 4 + 15) // 16 * 16}-byte row reads, 2e7 rows "
                                           "at random from an n_clusters-row array, L2 flushed "
                                           "(nr_measure_gather)",
                            "algorithmic_bytes_per_launch": sel_bytes,
                            "clusters_scored_per_query": st.scored / nq,
                            "avg_launch_ms": sel_avg_ms, "launches_per_step": n_ref},
        "stage_ms_per_step": {kk: v / args.steps for kk, v in stage_ms.items()},
        "e2e": {"value": e2e_v, "unit": "queries/s", "h2d_bytes_per_step": nq * row_bytes,
                "d2h_bytes_per_step": nq * k * 12},
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "setup_s": {"index_build": t_build, "ground_truth": t_gt},
        "index": {"builder": "gpu" if gpu_built else "host", "n_clusters": ix.n_clusters,
                  **({} if build_info is None else build_info)},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        if gpu_built:
            out["cpu_baseline"] = cpu_baseline_subindex(w, ix, qs, k, P, C, kw, args.cpu_seconds)
        else:
            cb, _ = cpu_baseline(w, path, qs, k, P, C, kw, args.cpu_seconds)
            out["cpu_baseline"] = cb
    if rank == 0:
        print(json.dumps(out), flush=True)
    ix.close()
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())

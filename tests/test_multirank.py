"""The benchmark's multi-rank host logic on the CPU, with two gloo ranks
(world size 2) as torchrun would start them: the job's time is its slowest
rank's, the job's throughput counts every rank's units, each rank searches its
own slice of one query stream, and the reference arm runs on rank 0 only.
Replicas share nothing on the data path, so this is all the N > 1 path adds."""
import json
import os
import socket

import numpy as np
import pytest

import bench
import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        local_ms = [12.5, 40.0][rank]          # rank 1 is the slow one
        job_ms = bench.max_over_ranks(local_ms, w)
        rate = bench.job_rate(10_000 * 5, w, job_ms / 1e3)
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"rank": r, "world": w, "local": local, "job_ms": job_ms, "rate": rate}, f)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(180)
def test_two_gloo_ranks_report_the_slowest_rank(tmp_path):
    import torch.multiprocessing as mp

    mp.spawn(_rank_main, args=(2, _free_port(), str(tmp_path)), nprocs=2, join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(2)]
    for r, d in enumerate(res):
        assert (d["rank"], d["world"], d["local"]) == (r, 2, r)
        assert d["job_ms"] == 40.0                       # max over ranks, on every rank
        assert d["rate"] == pytest.approx(2 * 10_000 * 5 / 0.040)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(7.25, 1) == 7.25
    assert bench.job_rate(100, 1, 0.5) == 200.0


def test_rank_query_batches_are_slices_of_one_stream():
    w = synth.WORKLOADS["tiny"]
    nq = 64
    both = synth.mixture(w, synth.SEED_QUERIES, 0, 2 * nq)
    r0 = synth.mixture(w, synth.SEED_QUERIES, 0 * nq, nq)
    r1 = synth.mixture(w, synth.SEED_QUERIES, 1 * nq, nq)
    assert np.array_equal(r0, both[:nq]) and np.array_equal(r1, both[nq:])
    assert np.array_equal(r0, synth.queries(w, nq))   # rank 0 searches the usual batch
    assert not np.array_equal(r0, r1)


def test_reference_arm_works_on_rank_zero_only():
    # any rank but 0 returns before reading its arguments
    assert bench.run_reference(None, None, 1, 2) == 0

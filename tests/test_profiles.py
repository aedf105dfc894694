"""The committed refine traffic record still describes the committed refine
kernel: bench.py reports ncu DRAM bytes only while the refine sources hash
to a capture's digest, so an edit to the kernel without a new capture would
silently drop the field to null. This fails first."""
import json
import os

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_refine_traffic_record_matches_the_refine_sources():
    rec = json.load(open(os.path.join(ROOT, "profiles", "refine_traffic.json")))
    digest = bench.refine_sources_digest()
    caps = rec["captures"]
    assert any(e["sources_sha256"] == digest for e in caps.values()), (
        "refine sources changed since the committed capture: re-capture the refine kernel "
        "(the command in profiles/refine_traffic.json) and record its digest")
    # the benchmark's workload is served (scaled from its proxy capture)
    by, src = bench.traffic_from_profile("u8-1b", 1024, 1024, 63.57e9)
    assert by is not None and src is not None and 0.9 < by / 63.57e9 < 1.2

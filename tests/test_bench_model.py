"""The measurement model of bench.py, checked on the CPU: the per-unit byte
model (written out by hand for a small hyperbatch), the launch count it
claims per step, and the lookup of the committed ncu traffic figure, which
must answer only for the profiled workload and the profiled gather source."""
import hashlib
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_algorithmic_bytes_by_hand():
    # two hops; |F_1| = 10, |F_2| = 25 (= |src_1|), |src_2| = rows = 60; int64 offsets
    c = {"frontier": [10, 25], "edges": [30, 70], "rows": 60, "distinct_rows": 40,
         "row_bytes": 256}
    got = bench.algorithmic_bytes(c, 8)
    hop1 = 10 * 2 * 8 + 30 * 4 + 30 * 4 + 10 * 8 + (25 - 10) * 4
    hop2 = 25 * 2 * 8 + 70 * 4 + 70 * 4 + 25 * 8 + (60 - 25) * 4
    gather = 60 * (256 + 8) + 40 * 256
    assert got == {"sampling": hop1 + hop2, "gather": gather, "total": hop1 + hop2 + gather}


def test_launch_count_per_step():
    # key + size fill, 4 for the targets, 16 per hop, mark + count + gather, one count per hop;
    # 60 at K = 3 is the count of the ncu launch list of one rmat100m hyperbatch
    assert bench.kernel_launches_per_step(3) == 60
    assert bench.kernel_launches_per_step(1) == 2 + 4 + 16 + 3 + 1


def test_profiled_traffic_only_for_its_workload_and_source():
    assert bench.gather_traffic_from_profile("rmat10m") is None
    src = os.path.join(ROOT, "paper_2601_01473_gb300", "csrc", "gather_hbm.cu")
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    profile = open(os.path.join(ROOT, "profiles", "gather_rmat100m.md")).read()
    t = bench.gather_traffic_from_profile("rmat100m")
    if f"gather_hbm.cu sha256 prefix: {sha}" in profile:
        assert t is not None and 1e9 < t < 1e11
    else:
        assert t is None

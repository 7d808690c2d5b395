"""bench.py's DRAM-traffic records (profiles/dram_traffic.json), on CPU.

The bench reports a kernel's ncu-measured DRAM bytes per launch only while
the hash of the kernel's sources equals the hash stored with the capture, so
a changed kernel never carries an old capture's figure.
"""

import hashlib
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

RECORDS = os.path.join(ROOT, "profiles", "dram_traffic.json")


def test_source_hash_is_the_sha256_of_the_named_sources():
    names = ("common.cuh", "kernels.h")
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2603_04427_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    assert bench.source_hash(*names) == h.hexdigest()[:16]
    assert bench.source_hash("kernels.h", "common.cuh") != bench.source_hash(*names)  # order counts


def test_a_record_is_reported_only_for_its_own_source_hash():
    with open(RECORDS) as f:
        d = json.load(f)
    for kernel, per_workload in d.items():
        if kernel.startswith("_"):
            continue
        for workload, e in per_workload.items():
            assert e["bytes_per_launch"] == e["read"] + e["write"]
            assert bench.recorded_traffic(kernel, workload, e["source_hash"]) == e["bytes_per_launch"]
            assert bench.recorded_traffic(kernel, workload, "0" * 16) is None
            assert "--clock-control none" in e["command"]
    assert bench.recorded_traffic("no_such_kernel", "x", "0" * 16) is None


def test_the_decode_record_is_close_to_the_algorithmic_bytes():
    """The headline decode moves K + V + q + out = 168.07 MB per launch; the
    committed capture must not show waste (re-reads) beyond a few percent."""
    with open(RECORDS) as f:
        e = json.load(f)["decode"]["mistral7b_gqa_decode_b16_ctx4096"]
    algorithmic = 16 * 8 * 4096 * (2 * 32 + 2 * 128) + 16 * 32 * 32 * 2 + 16 * 32 * 128 * 4
    assert algorithmic == 168067072
    assert 1.0 <= e["bytes_per_launch"] / algorithmic <= 1.05

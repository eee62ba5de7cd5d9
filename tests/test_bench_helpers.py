"""bench.py's tie between the committed ncu traffic record and the kernel
sources: the record is read only for the sources and the workload it was
captured on, and a comment or whitespace edit is not a kernel change."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_code_only_ignores_comments_and_whitespace():
    a = "int a = 1;  // the count\n/* a block\n comment */\nfloat b;\n"
    b = "int a=1;\n\n   float   b;"
    assert bench._code_only(a) == bench._code_only(b) == "inta=1;floatb;"
    assert bench._code_only("int a = 2;") != bench._code_only("int a = 1;")


def test_traffic_record_belongs_to_the_committed_kernels():
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        rec = json.load(f)["decode_partial"]
    assert rec["source_hash"] == bench._kernel_hash(), "decode kernel changed since its traffic capture"
    got = bench._ncu_traffic("decode_partial", rec["workload"])
    assert got == rec["dram_bytes_per_launch"]
    assert bench._ncu_traffic("decode_partial", "another_workload") is None
    assert bench._ncu_traffic("merge_prefill", rec["workload"]) is None

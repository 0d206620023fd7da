"""Host helpers of bench.py (CPU): the source hash that keys recorded ncu
traffic, and the recorded-traffic lookup."""
import json
import os
import sys

sys.path.insert(0, os.path.join(os.path.dirname(__file__), ".."))
import bench  # noqa: E402


def test_code_only_ignores_comments_and_blank_lines():
    a = "int f(int x) {\n  return x + 1;  // one more\n}\n"
    b = "/* the successor */\nint f(int x) {\n\n  return x + 1;\n}  // end\n"
    assert bench._code_only(a) == bench._code_only(b)


def test_code_only_sees_code_changes():
    a = "int f(int x) { return x + 1; }\n"
    b = "int f(int x) { return x + 2; }\n"
    assert bench._code_only(a) != bench._code_only(b)


def test_recorded_traffic_matches_the_current_sources():
    rec = json.load(open(os.path.join(os.path.dirname(__file__), "..", "profiles", "dram_traffic.json")))
    sha = bench.kernel_source_hash()
    for workload, ent in rec.items():
        got = bench.recorded_traffic(workload)
        if ent["kernel_sha"] == sha:
            assert got == ent["bytes_per_launch"] and got > 0
        else:
            assert got is None
    assert bench.recorded_traffic("no such workload") is None

"""Host-side pieces of bench.py that need no GPU: the algorithmic bytes of a
step, the workload description, and the key that ties a committed ncu figure
to the kernel code it measured."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads  # noqa: E402


def test_step_bytes_per_form():
    wl = workloads.workload("vgg16")
    assert bench.step_bytes(wl) == 12.0 * wl.K * wl.d  # read g, read e, write e
    assert bench.step_bytes(workloads.workload("vgg16_bf16")) == 10.0 * wl.K * wl.d
    loc = workloads.workload("vgg16_local")
    assert bench.step_bytes(loc) == 20.0 * loc.K * loc.d  # plus the momentum, read and written
    srv = workloads.workload("vgg16_alg3")
    assert bench.step_bytes(srv) == 12.0 * srv.K * srv.d + 20.0 * srv.d


def test_code_hash_ignores_comments_only():
    code = "int f(int x) {\n  return x + 1;  // one more\n}\n/* a note\n   over lines */\n"
    same = "// header\nint f(int x) {\n\n  return x + 1;\n}\n"
    other = "int f(int x) {\n  return x + 2;\n}\n"
    assert bench._code_only(code) == bench._code_only(same)
    assert bench._code_only(code) != bench._code_only(other)


def test_dram_summaries_name_their_code():
    """Every committed DRAM summary that bench.py reads gives its traffic per
    launch and the hash of the kernel code it was taken on (bench.py reports
    the traffic only while that code is current)."""
    import re
    for kernel, wl in [("accumulate", "vgg16"), ("accumulate", "resnet18"), ("rbgs_step", "resnet50")]:
        text = open(os.path.join(ROOT, "profiles", f"{kernel}_{wl}.md")).read()
        t = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
        h = re.search(r"source_hash:\s*([0-9a-f]{16})", text)
        assert t and h
        w = workloads.workload(wl)
        assert float(t.group(1)) >= 12.0 * w.K * w.d * 0.99  # at least the algorithmic bytes
    assert len(bench.kernel_source_hash()) == 16


def test_config_names_the_workload():
    import argparse
    wl = workloads.workload("resnet50")
    cfg = bench.config_of(wl, argparse.Namespace(gpus=1))
    assert cfg["d"] == wl.d and cfg["K"] == wl.K and cfg["compressor"] == "rbgs"
    assert cfg["block"] == wl.block and "resnet50" in cfg["workload"]

"""bench.py's reference arm (the fp64 oracle on the host cores) on CPU: one JSON line with
the contract's keys for the layer, backward, separable, IQBN and Poincare workloads."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

CASES = [
    (["--workload", "c1"], "TFLOP/s"),
    (["--workload", "c1", "--pass", "bwd"], "TFLOP/s"),
    ([], "images/s"),  # the default workload: the backbone
    (["--variant", "separable", "--workload", "c1"], "TFLOP/s"),
    (["--workload", "iqbn"], "images/s"),
    (["--workload", "poincare"], "images/s"),
]


@pytest.mark.parametrize("args,unit", CASES, ids=lambda a: ("_".join(a) or "default") if isinstance(a, list)
                         else None)
def test_reference_arm_json_line(args, unit):
    res = subprocess.run([sys.executable, "bench.py", "--impl", "reference", *args, "--steps",
                          "1", "--warmup", "1"], cwd=ROOT, capture_output=True, text=True,
                         timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1, res.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["unit"] == unit and d["value"] > 0 and d["higher_is_better"] is True
    assert d["steps"] == 1 and d["warmup"] == 1 and d["n_gpus"] == 1
    assert d["e2e"] == {"value": d["value"], "unit": unit, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert isinstance(d["config"]["workload"], str) and d["vs_baseline"] is None
    if not args:
        assert "backbone" in d["config"]["workload"]
    if "bwd" in args:
        assert "backward" in d["config"]["workload"]
    if "separable" in args:
        assert "Eq. 7" in d["config"]["workload"]


def test_workload_config_flops():
    from paper_2509_05512_gb300 import inputs
    full = bench.workload_config("c1", inputs)["flops_per_step"]
    assert bench.workload_config("c1", inputs, "separable")["flops_per_step"] == full / 4
    assert bench.workload_config("c1", inputs, "full", "bwd")["flops_per_step"] == 2 * full
    bb = bench.workload_config("backbone", inputs, act="silu")
    assert "SiLU" in bb["epilogue"] and bb["convs"] == 20


def test_recorded_traffic_lookup(tmp_path):
    # a record is used only for its own workload key, its own kernel (the library's full
    # name, template instance included) and the current device-code sources
    import json
    rec = {"c1": {"kernel": "qconv_ws_kernel<halo,issuers=2>", "dram_bytes_per_launch": 123,
                  "kernel_sha": bench.kernel_source_hash("qconv_ws_kernel<halo,issuers=2>")},
           "old": {"kernel": "qconv_ws_kernel<halo,issuers=2>", "dram_bytes_per_launch": 7,
                   "kernel_sha": "0000000000000000"}}
    path = str(tmp_path / "traffic.json")
    with open(path, "w") as f:
        json.dump(rec, f)
    assert bench.recorded_traffic("c1", "qconv_ws_kernel<halo,issuers=2>", path) == 123
    assert bench.recorded_traffic("c1", "qconv_ws_kernel<halo,issuers=3>", path) is None
    assert bench.recorded_traffic("c1", "qconv_tc_kernel<pair,kappa=32,bnq=64>", path) is None
    assert bench.recorded_traffic("old", "qconv_ws_kernel<halo,issuers=2>", path) is None
    assert bench.recorded_traffic("no_such_workload", None, path) is None

    # the hash follows the kernel's own sources: another kernel's file does not enter it
    assert bench.kernel_source_hash("qconv_ws_kernel<x>") != bench.kernel_source_hash(
        "qconv_vs_kernel<x>")
    assert bench.kernel_source_hash("qconv_ws_kernel<a>") == bench.kernel_source_hash(
        "qconv_ws_kernel<b>")
    assert bench.kernel_source_hash(None) == bench.kernel_source_hash("unknown_kernel")

    class A:
        workload, direction, variant = "c2a", "bwd", "separable"
    assert bench.traffic_key(A) == "c2a:bwd:sep"
    A.direction, A.variant = "fwd", "full"
    assert bench.traffic_key(A) == "c2a"


def test_kernel_sources_table_names_existing_files():
    # the traffic hash of a kernel covers the files of its KERNEL_SOURCES entry and the
    # shared headers: each must exist, or an edit to the kernel would go unnoticed
    import os
    csrc = os.path.join(bench.ROOT, "paper_2509_05512_gb300", "csrc")
    for kernel, files in bench.KERNEL_SOURCES.items():
        for name in files + bench.SHARED_DEVICE_SOURCES:
            assert os.path.isfile(os.path.join(csrc, name)), (kernel, name)
        assert name not in bench.HOST_ONLY_SOURCES
    # the dominant kernel of the default bench line has a record taken on its current
    # sources (the kernel name is the library's, without template arguments)
    import json
    with open(os.path.join(bench.ROOT, "profiles", "ncu_traffic.json")) as f:
        rec = json.load(f)["backbone"]
    assert rec["kernel"].split("<")[0] in bench.KERNEL_SOURCES

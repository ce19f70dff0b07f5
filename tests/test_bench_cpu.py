"""Parts of bench.py that need no GPU.

The DRAM traffic records behind roofline.traffic and kernels[*].dram_gb_s apply
only to the workload they were captured on and only while the kernel's sources
are unchanged.  The oracle arm (`--impl reference`) prints the contract's JSON
line, and fewer than three warm-up steps are refused."""
import hashlib
import json

import bench


def _write(tmp_path, workload, src_text, recorded_text):
    src = tmp_path / "kernel.cu"
    src.write_text(src_text)
    rec = {"about": "test", "workload": workload,
           "kernels": {"k": {"dram_bytes_per_launch_full_size": 1234.0,
                             "source_files": [str(src)],
                             "sources_sha256": hashlib.sha256(recorded_text.encode()).hexdigest()}}}
    path = tmp_path / "dram_traffic.json"
    path.write_text(json.dumps(rec))
    return str(path), src


def test_traffic_record_matches_workload_and_sources(tmp_path):
    path, _ = _write(tmp_path, "vitb_t17", "a", "a")
    assert bench.traffic_record("k", "vitb_t17", path) == 1234.0
    assert bench.traffic_record("k", "skew_t8", path) is None  # captured on another workload
    assert bench.traffic_record("other", "vitb_t17", path) is None  # no record


def test_traffic_record_stale_sources(tmp_path):
    path, src = _write(tmp_path, "vitb_t17", "a", "a")
    src.write_text("b")  # the kernel changed since the capture
    assert bench.traffic_record("k", "vitb_t17", path) is None


def test_committed_record_names_its_workload():
    with open(bench.os.path.join(bench.ROOT, "profiles", "dram_traffic.json")) as fh:
        rec = json.load(fh)
    assert rec["workload"] in bench.workloads.CONFIGS


def _run_bench(*args):
    import subprocess
    import sys
    return subprocess.run([sys.executable, bench.os.path.join(bench.ROOT, "bench.py"), *args],
                          capture_output=True, text=True, timeout=600)


def test_reference_arm_json_line():
    """The oracle arm the driver runs (`--impl reference`) prints one JSON line with
    the contract's keys; on the tiny workload it takes a couple of seconds."""
    r = _run_bench("--impl", "reference", "--config", "tiny_fp32", "--steps", "1", "--warmup", "3")
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["n_gpus"] == 1
    for key in ("metric", "unit", "steps", "warmup", "ms_per_step", "higher_is_better", "config"):
        assert key in line, key
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["e2e"]["value"] == line["value"]
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == line["value"]


def test_warmup_below_three_is_refused():
    r = _run_bench("--impl", "reference", "--config", "tiny_fp32", "--steps", "1", "--warmup", "2")
    assert r.returncode != 0 and "--warmup" in r.stderr

"""Host logic of bench.py that needs no GPU: the DRAM traffic records behind
roofline.traffic and kernels[*].dram_gb_s apply only to the workload they were
captured on and only while the kernel's sources are unchanged."""
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

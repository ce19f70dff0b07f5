"""Parts of bench.py that need no GPU.

The DRAM traffic records behind roofline.traffic and kernels[*].dram_gb_s are
one-kernel ncu captures on a prefix of a workload's tasks, scaled to the full
workload by the algorithmic bytes; they apply only to the workload they were
captured on and only while the kernel's sources are unchanged.  L2 is flushed
between timed steps for the workloads whose weights are small against L2.  The oracle arm (`--impl reference`) prints the contract's JSON
line, and fewer than three warm-up steps are refused."""
import hashlib
import json

import bench


def _write(tmp_path, workload, src_text, recorded_text):
    src = tmp_path / "kernel.cu"
    src.write_text(src_text)
    rec = {"about": "test",
           "workloads": {workload: {"tasks": 2, "kernels": {"k": {
               "dram_bytes_per_launch": 1200, "algorithmic_bytes_per_launch": 1000,
               "source_files": [str(src)],
               "sources_sha256": hashlib.sha256(recorded_text.encode()).hexdigest()}}}}}
    path = tmp_path / "dram_traffic.json"
    path.write_text(json.dumps(rec))
    return str(path), src


def test_traffic_record_scales_prefix_capture(tmp_path):
    """A prefix capture of 1200 DRAM bytes for 1000 algorithmic bytes gives 1.2x
    the full launch's algorithmic bytes."""
    path, _ = _write(tmp_path, "vitb_t17", "a", "a")
    assert bench.traffic_record("k", "vitb_t17", 1000, path) == 1200.0
    assert bench.traffic_record("k", "vitb_t17", 8500, path) == 10200.0
    assert bench.traffic_record("k", "skew_t8", 1000, path) is None  # captured on another workload
    assert bench.traffic_record("other", "vitb_t17", 1000, path) is None  # no record


def test_traffic_record_stale_sources(tmp_path):
    path, src = _write(tmp_path, "vitb_t17", "a", "a")
    src.write_text("b")  # the kernel changed since the capture
    assert bench.traffic_record("k", "vitb_t17", 1000, path) is None


def test_write_traffic_record_round_trip(tmp_path):
    """The writer reads ncu's --csv log and the plain run's JSON line; the record
    then reads back through traffic_record with the sources as they are now."""
    plain = tmp_path / "plain.json"
    plain.write_text(json.dumps({"kernels": {"tc_dw1": {"algorithmic_bytes_per_launch": 1000}}}) + "\n")
    log = tmp_path / "dw1.csv"
    log.write_text('==PROF== Connected\n'
                   '"ID","Kernel Name","Metric Name","Metric Unit","Metric Value"\n'
                   '"0","wgrad_pair_kernel","dram__bytes_read.sum","Mbyte","1.5"\n'
                   '"0","wgrad_pair_kernel","dram__bytes_write.sum","byte","500"\n')
    out = tmp_path / "rec.json"
    bench.write_traffic_record("vitb_t17", 2, str(plain), [("tc_dw1", str(log))], path=str(out))
    rec = json.loads(out.read_text())["workloads"]["vitb_t17"]
    assert rec["kernels"]["tc_dw1"]["captured_at_tasks"] == 2
    assert rec["kernels"]["tc_dw1"]["dram_bytes_per_launch"] == 1500500
    assert bench.traffic_record("tc_dw1", "vitb_t17", 2000, str(out)) == 3001000.0


def test_committed_record_names_known_workloads_and_kernels():
    with open(bench.os.path.join(bench.ROOT, "profiles", "dram_traffic.json")) as fh:
        rec = json.load(fh)
    for wl, entry in rec["workloads"].items():
        assert wl in bench.workloads.CONFIGS
        for name, k in entry["kernels"].items():
            assert name in bench.KERNEL_SOURCES
            # a prefix of the tasks, or the full size (one-pass DRAM counters only)
            assert 1 <= k["captured_at_tasks"] <= bench.workloads.CONFIGS[wl].T


def test_l2_policy():
    """L2 is flushed between timed steps where the weights are small against L2
    (ViT-S 4 tasks, ViT-B 6 tasks), not where they are 40x it (ViT-B 17 tasks)."""
    cf = bench.workloads.CONFIGS
    assert bench.l2_policy(cf["vits_t4"])[0] and bench.l2_policy(cf["vitb_t6"])[0]
    assert not bench.l2_policy(cf["vitb_t17"])[0] and not bench.l2_policy(cf["skew_t8"])[0]
    assert "5.13 GB" in bench.l2_policy(cf["vitb_t17"])[1]


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

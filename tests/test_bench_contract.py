"""bench.py's JSON line: the keys and types the benchmark contract requires,
for the reference arm (the oracle on the host; runs on CPU) and, on a GB300,
for the library's own arm on a small workload."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args, timeout=600):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                       cwd=ROOT, capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


def _common(d):
    for k, t in (("metric", str), ("value", float), ("unit", str),
                 ("n_gpus", int), ("steps", int), ("warmup", int),
                 ("higher_is_better", bool), ("scaling", str), ("dtype", str),
                 ("data", str), ("config", dict)):
        assert isinstance(d[k], t), k
    assert d["vs_baseline"] is None  # the paper reports no number for this path
    assert d["config"]["workload"]
    assert "model" not in d["config"]
    assert d["value"] > 0
    assert d["scaling"] == "weak" and d["higher_is_better"] is True


def test_reference_arm_line():
    d = _run("--impl", "reference", "--steps", "1", "--warmup", "1")
    _common(d)
    assert d["impl"] == "reference"
    assert d["dtype"] == "f64"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"],
                        "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


@pytest.mark.gpu
def test_gpu_arm_line():
    d = _run("--workload", "480p", "--steps", "3", "--warmup", "3",
             "--cpu-seconds", "2", "--no-per-workload")
    _common(d)
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3
    assert d["dtype"] == "bf16"
    assert d["ms_per_step"] > 0
    r = d["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert 0 < r["frac"] <= 1.2 and abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] > 0
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    # one append, one attention call and at most one merge per chunk and step
    assert 2 * 8 * 3 <= d["gpu_launches"] <= 3 * 8 * 3
    c = d["clocks"]
    assert c["sm_max_mhz"] > 0 and isinstance(c["reasons"], list)


def test_traffic_is_reported_only_for_the_profiled_source(tmp_path, monkeypatch):
    """The roofline's `traffic` comes from a committed ncu summary only while
    the kernel source it was taken on is unchanged (else null)."""
    import hashlib
    sys.path.insert(0, ROOT)
    import bench
    src = tmp_path / "paper_2609_36757_gb300" / "csrc" / "k.cu"
    src.parent.mkdir(parents=True)
    src.write_bytes(b"__global__ void k() {}\n")
    prof = tmp_path / "profiles"
    prof.mkdir()
    digest = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (prof / "k_case_traffic.txt").write_text(
        "# comment = ignored\nsource=k.cu\nsource_sha256_16=%s\n"
        "dram_bytes_capture=10\ndram_bytes_per_avg_launch=12345\n" % digest)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_traffic("k_case") == 12345.0
    assert bench.load_traffic("missing_case") is None
    src.write_bytes(b"__global__ void k() { /* changed */ }\n")
    assert bench.load_traffic("k_case") is None


@pytest.mark.gpu
def test_per_workload_leg_keys():
    """One per-workload leg (the tiny stream): the keys the bench line
    carries for each stream of the metric."""
    sys.path.insert(0, ROOT)
    import torch
    import bench
    from paper_2609_36757_gb300 import workloads as WL
    peaks, _ = bench.load_peaks()
    leg = bench.measure_workload(WL.TINY, torch.device("cuda", 0), peaks, 0,
                                 steps=2, warmup=1)
    assert leg["steps"] == 2 and leg["warmup"] == 1
    assert leg["flops_per_step"] > 0
    for k in ("path_tflops", "kernel_tflops", "latent_frames_per_s",
              "kernel_frac_of_sustained", "kernel_frac_of_burst"):
        assert leg[k] > 0, k
    assert leg["kernel_tflops"] >= leg["path_tflops"] * 0.5
    assert set(leg["ms_per_chunk"]) == {"mean_fwd", "last_fwd",
                                        "mean_step_per_chunk"}
    assert leg["gpu_launches"] >= 2 * WL.TINY.num_chunks * 2
    assert leg["shape"]["chunks"] == WL.TINY.num_chunks


def test_append_dram_is_reported_only_for_the_profiled_source(tmp_path,
                                                             monkeypatch):
    """The append's DRAM-seen bytes come from a committed ncu summary only
    while the append kernel source is unchanged (else null)."""
    import hashlib
    sys.path.insert(0, ROOT)
    import bench
    src = tmp_path / "paper_2609_36757_gb300" / "csrc" / "kv_append.cu"
    src.parent.mkdir(parents=True)
    src.write_bytes(b"// append\n")
    prof = tmp_path / "profiles"
    prof.mkdir()
    digest = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (prof / "kv_append_1080p_traffic.txt").write_text(
        "source=kv_append.cu\nsource_sha256_16=%s\n"
        "algorithmic_read_bytes=100\nalgorithmic_write_bytes=100\n"
        "dram_read_bytes=100\ndram_write_bytes_during_launch=40\n"
        "ncu_time_ns=1000\n" % digest)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    d = bench.append_dram({"hbm_gbs": 1000.0})
    assert d["read_bytes"] == 100 and d["write_bytes_during_launch"] == 40
    assert abs(d["dram_gbs_during_launch"] - 140.0 / 1000e-9 / 1e9) < 1e-9
    assert abs(d["dram_frac_of_hbm"] - d["dram_gbs_during_launch"] / 1000.0) < 1e-12
    src.write_bytes(b"// changed\n")
    assert bench.append_dram({"hbm_gbs": 1000.0}) is None


@pytest.mark.gpu
def test_train_leg_keys():
    """The training-form leg of the default line (forward + backward of one
    one-shot sequence), on a small d = 128 sequence: keys and consistency of
    the rates with the times."""
    sys.path.insert(0, ROOT)
    import torch
    import bench
    from paper_2609_36757_gb300 import workloads as WL
    peaks, _ = bench.load_peaks()
    w = WL.Workload("train-small", 1, 4, 128, 256, 2, 3, window_chunks=1,
                    seed=11)
    leg = bench.measure_train_leg(w, torch.device("cuda", 0), peaks, 0,
                                  steps=2, warmup=1)
    assert leg["steps"] == 2 and leg["warmup"] == 1
    assert leg["bwd_flops"] == 2.5 * leg["fwd_flops"] > 0
    for k in ("fwd_ms", "bwd_ms", "fwd_tflops", "bwd_tflops",
              "fwd_frac_of_burst", "bwd_frac_of_burst"):
        assert leg[k] > 0, k
    assert abs(leg["bwd_tflops"] - leg["bwd_flops"] / leg["bwd_ms"] / 1e9) < 1e-6 * leg["bwd_tflops"]
    assert leg["shape"]["tokens"] == w.num_tokens

"""Host-side logic of bench.py that needs no GPU: the roofline denominators,
the committed traffic figure and its source check, and the reference arm's
JSON line (the oracle on the host cores)."""
import json
import os
import subprocess
import sys

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_measured_peak_is_read_from_the_peaks_file():
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        want = float(json.load(f)["hbm_gbs"])
    assert bench.measured_peaks() == (want, "measured")


def test_missing_peaks_file_gives_the_fallback(monkeypatch, tmp_path):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.measured_peaks() == (bench.FALLBACK_HBM_GBS, "fallback")


def test_committed_traffic_follows_the_kernel_source(monkeypatch):
    import re
    name = "llama3-8b-bf16-per-tensor"
    text = open(os.path.join(ROOT, "profiles", "k_hash_probe.%s.md" % name)).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)\s+source_digest:\s*([0-9a-f]+)",
                  text)
    assert m, "the profile summary carries no traffic line"
    # the figure is reported exactly while the kernel source is the one it was
    # taken on (the digest in the summary), and dropped for any other source
    monkeypatch.setattr(bench, "kernel_source_digest", lambda: m.group(2))
    traffic = bench.committed_traffic(name)
    assert traffic == float(m.group(1)) and traffic > 16.06e9
    assert bench.committed_traffic("no-such-workload") is None
    monkeypatch.setattr(bench, "kernel_source_digest", lambda: "0" * 16)
    assert bench.committed_traffic(name) is None  # changed source: no figure


def test_kernel_source_digest_covers_the_hash_kernel_sources(monkeypatch, tmp_path):
    d0 = bench.kernel_source_digest()
    fake = tmp_path / "paper_2607_23115_gb300" / "csrc"
    fake.mkdir(parents=True)
    src = os.path.join(ROOT, "paper_2607_23115_gb300", "csrc")
    for f in os.listdir(src):
        if f.endswith((".cu", ".cuh")):
            (fake / f).write_bytes(open(os.path.join(src, f), "rb").read())
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.kernel_source_digest() == d0
    p = fake / "staged_hash.cuh"
    p.write_bytes(p.read_bytes() + b"\n")
    assert bench.kernel_source_digest() != d0


@pytest.mark.timeout(600)
def test_reference_arm_prints_one_line_on_the_host_cores():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload",
                          "fp16-64m", "--steps", "2", "--warmup", "3"],
                         cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["metric"] == bench.METRIC
    assert j["unit"] == "GB/s" and j["higher_is_better"] is True
    assert j["steps"] == 2 and j["warmup"] == 3 and j["value"] > 0
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["cores"] == 1
    assert j["cpu_baseline"]["value"] == j["value"]
    assert j["e2e"] == {"value": j["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert j["config"]["workload"] == "fp16-64mib-half-prefilled"
    # the same config object as the GPU arm's
    assert set(j["config"]) == {"workload", "description", "payload_bytes_per_step",
                                "payloads_per_step", "chunk_bytes", "chunks_per_step",
                                "misses_per_step", "cache_capacity_bytes", "key16",
                                "paper_ids", "evict_lru"}
    assert j["config"]["misses_per_step"] == 8192

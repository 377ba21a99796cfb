"""bench.py's reference arm (the oracle on the host cores) prints one JSON
line with the contract's keys; it needs no GPU."""
import json
import os
import subprocess
import sys

from conftest import ROOT


def test_reference_arm_json_line():
    env = dict(os.environ, RANK="0")
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--config", "k7_r3_d4096_alie", "--steps", "1", "--warmup", "0"],
                       capture_output=True, text=True, timeout=300, env=env, cwd=ROOT)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in j, key
    assert j["impl"] == "reference" and j["unit"] == "ms/round" and j["value"] > 0
    assert j["higher_is_better"] is False
    assert j["config"]["workload"] == "k7_r3_d4096_alie"
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["cores"] >= 1
    assert j["e2e"]["h2d_bytes_per_step"] == 0 and j["e2e"]["value"] == j["value"]


def test_profile_traffic_lines_parse_and_scale(tmp_path, monkeypatch):
    """The roofline's `traffic` comes from a committed ncu summary: the line
    is found, scaled by the units processed, and ignored once the kernel's
    source no longer has the recorded hash."""
    import hashlib
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    src = tmp_path / "k.cu"
    src.write_text("// kernel\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "k.md").write_text(
        f"text\nbench-traffic: my_kernel workload=w@d=1 units=100 dram_bytes=250 source_sha={sha}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profile_traffic("my_kernel", "w", 400, str(src)) == 1000
    assert bench.profile_traffic("other_kernel", "w", 400, str(src)) is None
    src.write_text("// kernel, changed\n")
    assert bench.profile_traffic("my_kernel", "w", 400, str(src)) is None


def test_committed_profiles_carry_traffic_lines():
    """Every kernel the bench line reports traffic for has a summary line."""
    text = "".join(open(os.path.join(ROOT, "profiles", fn)).read()
                   for fn in os.listdir(os.path.join(ROOT, "profiles")) if fn.endswith(".md"))
    for tag in ("compare_vec_kernel", "aggregate_kernel"):
        assert f"bench-traffic: {tag} " in text, tag

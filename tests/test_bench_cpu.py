"""bench.py on CPU: workload presets and the oracle reference arm's JSON line."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_workload_layers_exceed_l2(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    for name, w in bench.WORKLOADS.items():
        monkeypatch.setattr(sys, "argv", ["bench.py", "--workload", name])
        a = bench.parse_args()
        e = 4 if a.w["dtype"] == "f32" else 2
        per_layer = a.w["N"] * (a.w["Hq"] + 2 * a.w["Hkv"]) * a.w["D"] * e
        assert a.w["layers"] * per_layer >= bench.L2_FLUSH_BYTES, name
        cfg = bench.workload_config(a)
        assert cfg["name"] == name and cfg["workload"].startswith(name)
    monkeypatch.setattr(sys, "argv", ["bench.py"])
    a = bench.parse_args()
    assert a.w["name"] == "C5" and a.w["layers"] == 28 and a.w["N"] == 65536
    assert [r[:2] for r in a.w["runs"]] == [("stochastic", 0), ("structural", 1)]


def test_reference_arm_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "C1",
                        "--steps", "1", "--warmup", "1", "--cpu-seconds", "1"],
                       capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["unit"] == "pair-heads/s"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["config"]["name"] == "C1" and line["higher_is_better"] is True


def test_recorded_traffic_follows_the_source_hashes(monkeypatch, tmp_path):
    """The DRAM bytes recorded under profiles/traffic.json count only while every kernel source
    they were captured on is unchanged (sha256 prefix); a changed source gives no traffic."""
    import hashlib

    sys.path.insert(0, ROOT)
    import bench

    csrc = tmp_path / "paper_2607_21927_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    (csrc / "a.cu").write_text("kernel a\n")
    (csrc / "b.cu").write_text("kernel b\n")
    h = {n: hashlib.sha256((csrc / n).read_bytes()).hexdigest()[:16] for n in ("a.cu", "b.cu")}
    rec = {"a.cu": {"W": {"source_sha256_16": h["a.cu"], "dram_bytes_per_launch_full_size": 123}},
           "a.cu+b.cu": {"W": {"source_sha256_16": [h["a.cu"], h["b.cu"]], "dram_bytes_per_launch_full_size": 456}}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.recorded_traffic(("a.cu",), "W") == 123
    assert bench.recorded_traffic(("a.cu", "b.cu"), "W") == 456
    assert bench.recorded_traffic(("a.cu",), "other") is None
    (csrc / "b.cu").write_text("kernel b, edited\n")
    assert bench.recorded_traffic(("a.cu", "b.cu"), "W") is None
    assert bench.recorded_traffic(("a.cu",), "W") == 123

"""bench.py's reference arm (the float64 oracle on the host cores) and its
JSON contract, on the CPU."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "3",
                        "--warmup", "3", "--workload", "tiny"], capture_output=True, text=True, timeout=600,
                       cwd=ROOT)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in j, key
    assert j["impl"] == "reference" and j["value"] > 0 and j["higher_is_better"] is True
    assert j["config"]["workload"] == "tiny" and "l2" in j["config"]
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["value"] == j["value"]
    assert j["e2e"]["h2d_bytes_per_step"] == 0 and j["e2e"]["d2h_bytes_per_step"] == 0


def test_warmup_below_three_is_refused():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--warmup", "1"],
                       capture_output=True, text=True, timeout=120, cwd=ROOT)
    assert r.returncode != 0


def test_sweep_names_resolve():
    from paper_2506_08520_gb300 import sweep, workloads
    for name in sweep.DEFAULT:
        assert name in workloads.WORKLOADS or name in sweep.MIXES, name
    for parts in sweep.MIXES.values():
        assert all(p in workloads.WORKLOADS for p in parts)


def test_sweep_list_runs_without_a_gpu(capsys):
    from paper_2506_08520_gb300 import sweep
    assert sweep.main(["--list", "uformer-mix", "tiny"]) == 0
    assert capsys.readouterr().out.split() == ["uformer-mix", "tiny"]


def test_reference_arm_of_the_fused_projection_workload():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "3",
                        "--warmup", "3", "--workload", "uformer-s4-qkv"], capture_output=True, text=True,
                       timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    j = json.loads([l for l in r.stdout.splitlines() if l.startswith("{")][-1])
    assert j["impl"] == "reference" and j["value"] > 0
    assert j["config"]["workload"] == "uformer-s4-qkv" and "front" in j["config"]
    assert "projections made beforehand" in j["cpu_baseline"]["sample"]


def test_unit_flops_counts_the_projection():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2506_08520_gb300 import workloads
    wl = workloads.WORKLOADS["swinir256-bf16"]
    fused = workloads.WORKLOADS["swinir256-bf16-qkv"]
    assert bench.unit_flops(fused) - bench.unit_flops(wl) == 2 * 64 * 180 * 90
    assert fused.io_bytes == (2 * 1024 * 64 * 180 + 3 * 180 * 180) * 2

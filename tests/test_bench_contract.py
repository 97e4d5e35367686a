"""bench.py's reference arm (the CPU oracle) prints one JSON line with the contract's keys
(CPU only; a tiny sample of the workload)."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_contract_line():
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
           "--warmup", "0", "--config", "g8_t1k_d2048_v32k", "--ref-tokens", "4"]
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "impl",
              "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["config"]["workload"] == "g8_t1k_d2048_v32k"


def test_gpus_flag_launches_one_process_per_gpu():
    """`bench.py --gpus 2` without a torch.distributed environment re-launches itself under
    torch.distributed.run with two ranks (127.0.0.1 rendezvous); for the reference arm rank 0
    alone prints the line, with n_gpus = 2, and the other rank exits 0."""
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
           "--steps", "1", "--warmup", "0", "--config", "g8_t1k_d2048_v32k", "--ref-tokens", "2",
           "--master-port", "29541"]
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [json.loads(x) for x in out.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    assert lines[0]["n_gpus"] == 2 and lines[0]["impl"] == "reference"
    assert lines[0]["cpu_baseline"]["cores"] >= 1


def test_traffic_figure_is_keyed_to_kernel_source_and_tile_mode(tmp_path, monkeypatch):
    """The roofline's `traffic` comes from a committed ncu summary only if that summary was taken
    on the current GEMM source in the tile mode the kernel runs in now (a summary without a
    tile_mode line counts as single-CTA tiles); the committed full-size summaries carry the
    three keys."""
    sys.path.insert(0, ROOT)
    import bench
    import re
    wl = "g16_t16k_d5120_v152k"
    for kernel in bench.GEMM_KERNELS:
        txt = open(os.path.join(ROOT, "profiles", f"{kernel}__{wl}.md")).read()
        for key in ("source_sha", "tile_mode", "dram_bytes_per_launch_full"):
            assert re.search(key + r":\s*\S+", txt), (kernel, key)
    sha = bench.kernel_source_sha()
    monkeypatch.setattr(bench, "PROFILES", str(tmp_path))
    (tmp_path / "k__w.md").write_text(
        f"source_sha: {sha}\ntile_mode: 4\ndram_bytes_per_launch_full: 1.5e+12\n")
    (tmp_path / "k0__w.md").write_text(f"source_sha: {sha}\ndram_bytes_per_launch_full: 2e+11\n")
    (tmp_path / "old__w.md").write_text(
        "source_sha: 0000000000000000\ntile_mode: 0\ndram_bytes_per_launch_full: 2e+11\n")
    assert bench.ncu_traffic("k", "w", 4) == 1.5e12
    assert all(bench.ncu_traffic("k", "w", m) is None for m in (0, 1, 2, 3))
    assert bench.ncu_traffic("k0", "w", 0) == 2e11 and bench.ncu_traffic("k0", "w", 2) is None
    assert bench.ncu_traffic("old", "w", 0) is None
    assert bench.ncu_traffic("missing", "w", 0) is None

"""Host-side logic of bench.py, checked without a GPU: the algorithmic work it divides by the
measured times, the roofline arithmetic, the shared workload config of both arms, and the
argument defaults the timing rules ask for."""
import importlib.util
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_defaults_follow_the_timing_rules(bench):
    a = bench.parse_args([])
    assert a.gpus == 1 and a.warmup >= 3 and a.steps >= 1 and a.impl == "ilw"
    assert bench.parse_args(["--impl", "reference"]).impl == "reference"


def test_kernel_work_of_the_medium_backbone(bench):
    """Per launch at 8 images of 1600 tokens, d 384, 6 heads, MLP 1536: 2 M N K operations per GEMM
    (M = 12800 tokens), scores B H T^2 for global attention and B H 4 (T/4)^2 for 2x2 windows, and
    3 bytes per I-LayerNorm element (int16 in, the int8 value out in one byte)."""
    cfg = bench.workload_cfg()
    assert (cfg["B"], cfg["T"], cfg["d"], cfg["H"], cfg["F"], cfg["layers"]) == (8, 1600, 384, 6, 1536, 10)
    w = bench.kernel_work(cfg, cfg["B"])
    M = 8 * 1600
    assert w["gemm_qkv"] == ("tensor", 2.0 * M * 1152 * 384)
    assert w["gemm_proj"] == ("tensor", 2.0 * M * 384 * 384)
    assert w["gemm_fc1_gelu"] == ("tensor", 2.0 * M * 1536 * 384)
    assert w["gemm_fc2"] == ("tensor", 2.0 * M * 384 * 1536)
    assert w["patch_embed"] == ("tensor", 2.0 * M * 384 * 3 * 16 * 16)
    assert w["attention_global"] == ("alu", 122_880_000.0)
    assert w["attention_window"] == ("alu", 8 * 6 * 4 * 400 * 400.0)
    assert w["layernorm"] == ("hbm", 3.0 * M * 384)


def test_roofline_entries(bench):
    peaks = {"hbm_gbs": 6670.9, "bf16_tflops_sustained": 1736.0}
    clocks = {"sm_mhz": 2070.0}
    k = {"avg_ms": 0.2}
    alu = bench.roofline_entry("attention_global", k, ("alu", 122.88e6), peaks, clocks, 152)
    peak = 152 * 128 * 2070e6 / 1e12
    assert alu["bound"] == "alu" and alu["peak"] == pytest.approx(peak)
    assert alu["achieved"] == pytest.approx(122.88e6 * 35 / 0.2e-3 / 1e12)
    assert alu["frac"] == pytest.approx(alu["achieved"] / peak)
    assert alu["frac_at_16_ops_per_score"] == pytest.approx(alu["frac"] * 16 / 35)
    hbm = bench.roofline_entry("layernorm", {"avg_ms": 0.011}, ("hbm", 3.0 * 12800 * 384), peaks, clocks, 152)
    assert hbm["unit"] == "GB/s" and hbm["peak"] == 6670.9
    assert hbm["achieved"] == pytest.approx(3.0 * 12800 * 384 / 0.011e-3 / 1e9)
    ten = bench.roofline_entry("gemm_fc2", {"avg_ms": 0.0244}, ("tensor", 2.0 * 12800 * 384 * 1536), peaks, clocks, 152)
    assert ten["unit"] == "TFLOP/s" and ten["frac"] == pytest.approx(ten["achieved"] / 1736.0)
    for e in (alu, hbm, ten):
        assert set(e) >= {"bound", "achieved", "peak", "unit", "frac", "traffic"}


def test_both_arms_report_one_config(bench):
    """The GPU arm and the reference arm take their `config` from the same function, which names
    the workload and the L2 policy and carries no model keys."""
    cfg = bench.workload_cfg()
    c = bench.workload_config(cfg, 1)
    assert c["workload"].startswith("medium_backbone_b8") and c["B"] == 8 and c["T"] == 1600 and "l2" in c
    assert "model" not in c
    assert bench.workload_config(cfg, 4)["parallelism"] == "replicas x4"


def test_reference_arm_prints_one_contract_line():
    """`bench.py --impl reference` (the oracle on the host's cores) prints one JSON line with the
    metric, unit and config of the GPU arm, its own CPU baseline and a zero-copy e2e block."""
    import json
    import subprocess
    import sys

    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["unit"] == "block-tokens/s" and line["value"] > 0
    assert line["higher_is_better"] is True and line["steps"] == 1 and line["warmup"] == 0
    assert line["config"]["workload"].startswith("medium_backbone_b8")
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"] and cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_reference_arm_runs_on_rank_zero_only():
    """Under torchrun the reference arm runs and prints on rank 0 alone; another rank exits 0
    without work or output."""
    import subprocess
    import sys

    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=300, cwd=ROOT,
                       env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    assert not [ln for ln in r.stdout.splitlines() if ln.startswith("{")]

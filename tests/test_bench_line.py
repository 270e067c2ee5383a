"""The benchmark's JSON line (bench.make_line) from fixed measured
quantities: every key of the benchmark contract is present with the
documented meaning, and the derived numbers follow from the inputs.  CPU
only."""
import json

import pytest

import bench


def _measured(**kw):
    m = dict(workload="4b-b1", shape_name="4b", dtype="bf16", n_gpus=1, steps=100, warmup=5, batch=2,
             prompt_tokens=2048, ms=250.0, ms_all=260.0, tokens=260, tokens_all=260, ctx_avg=1074.5, tau=0.5,
             force=0, prefill_s=3.0, prefill_rows=0, sampler=False, desc="B=2 projections=...",
             fam={0: {"bytes": 8.0e9, "ms": 2.0, "launches": 150, "replays": 64},
                  1: {"bytes": 1.0e8, "ms": 0.4, "launches": 37, "replays": 64}}, hbm=6774.6,
             peak_source="measured", step_bytes=9.3e9, cpu={"value": 5.0, "unit": "tokens/s", "cores": 16,
                                                             "kind": "oracle", "sample": "1 step"},
             e2e_s=30.0, e2e_tokens=240, launches=192, clocks={"sm_mhz": 2070, "sm_max_mhz": 2070, "reasons": []},
             regular=None)
    m.update(kw)
    return m


def test_contract_keys_and_meanings():
    line = bench.make_line(_measured())
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert k in line, k
    assert line["value"] == pytest.approx(260 / 0.260)          # all tokens / slowest rank's time
    assert line["ms_per_step"] == pytest.approx(2.6)
    assert line["higher_is_better"] is True and line["scaling"] == "weak" and line["vs_baseline"] is None
    assert line["config"]["workload"] == "4b-b1"
    assert line["config"]["acceptance"] == pytest.approx(260 / (100 * 2) - 1)
    r = line["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in r, k
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 6774.6
    assert r["achieved"] == pytest.approx(8.0e9 / 2.0e-3 / 1e9)  # family bytes / family time
    assert r["frac"] == pytest.approx(r["achieved"] / 6774.6)
    assert r["algorithmic_bytes_per_launch"] == pytest.approx(8.0e9 / 150)
    assert r["avg_launch_us"] == pytest.approx(2000.0 / 150)
    # the family's replay time is part of the step: its share is at most 1
    assert r["family_share_of_step"] == pytest.approx(2.0 / 2.5) and r["family_share_of_step"] <= 1.0
    assert r["launches_per_step"] * r["avg_launch_us"] <= 1e3 * line["ms_per_step"]
    assert r["attention"]["achieved"] == pytest.approx(1.0e8 / 0.4e-3 / 1e9)
    assert r["traffic"] is None
    assert r["step"]["achieved"] == pytest.approx(9.3e9 / 2.5e-3 / 1e9)
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 16
    e = line["e2e"]
    assert e["value"] == pytest.approx(8.0) and e["h2d_bytes_per_step"] == 16 and e["d2h_bytes_per_step"] == 24
    assert line["gpu_launches"] == 192 * 100
    json.dumps(line)  # serialisable


def test_regular_ratios():
    reg = dict(ms_per_step=2.0, ms_per_token=2.0, tokens_per_s=500.0, achieved_gbs=4000.0, prefill_s=6.0,
               pipo_prefill_warm_s=2.0)
    line = bench.make_line(_measured(regular=reg))
    # the pair step: 2.5 ms per step, 1.3 tokens per sequence and step
    assert line["regular"]["tpot_ratio"] == pytest.approx(2.0 / (2.5 / 1.3))
    assert line["regular"]["ttft_ratio"] == pytest.approx(3.0)
    assert line["regular"]["frac"] == pytest.approx(4000.0 / 6774.6)


def test_prefill_tensor_fraction():
    """The time to first token against the prefill's multiply-add flops and
    the measured bf16 peak; absent when either is unknown."""
    line = bench.make_line(_measured(prefill_flops=1.5e14, bf16_tflops=1934.6))
    pf = line["prefill"]
    assert pf["achieved_tflops"] == pytest.approx(1.5e14 / 3.0 / 1e12)
    assert pf["frac"] == pytest.approx(50.0 / 1934.6) and pf["bound"] == "tensor"
    assert pf["pair_positions"] == 1024 and pf["seconds"] == 3.0
    assert "prefill" not in bench.make_line(_measured())
    assert "prefill" not in bench.make_line(_measured(prefill_flops=1.5e14, bf16_tflops=None))


def test_missing_family_time_gives_no_fraction():
    line = bench.make_line(_measured(fam={0: {"bytes": 0.0, "ms": 0.0, "launches": 0, "replays": 0},
                                          1: {"bytes": 0.0, "ms": 0.0, "launches": 0, "replays": 0}}))
    assert line["roofline"]["achieved"] is None and line["roofline"]["frac"] is None


def test_recorded_traffic_needs_the_current_sources(tmp_path):
    from paper_2605_27255_gb300 import roofline
    csrc = tmp_path / "csrc"
    csrc.mkdir()
    (csrc / "k.cuh").write_text("kernel v1")
    prof = tmp_path / "profiles"
    prof.mkdir()
    d = roofline.sources_digest(str(csrc))
    (prof / "x.md").write_text(f"# summary\ntraffic: workload=9b-b8 bytes_per_launch=1.5e8 sources={d}\n")
    t = roofline.recorded_traffic(str(prof), "9b-b8", str(csrc))
    assert t["bytes_per_launch"] == 1.5e8 and t["source"].startswith("profiles/x.md")
    assert roofline.recorded_traffic(str(prof), "4b-b1", str(csrc)) is None
    (csrc / "k.cuh").write_text("kernel v2")  # the kernels changed since the capture
    assert roofline.recorded_traffic(str(prof), "9b-b8", str(csrc)) is None
    line = bench.make_line(_measured(traffic=t))
    assert line["roofline"]["traffic"] == 1.5e8


def test_reference_arm_runs_on_cpu_and_prints_one_contract_line():
    """bench.py --impl reference on the tiny workload (the fp64 oracle on the
    host cores): exit 0 and one JSON line with the reference arm's keys."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["steps"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}

"""bench.py pieces that need no GPU: the reference arm (the fp64 oracle timed on the
host cores), the parsing of the clock record taken during the timed region, the code
hash that keys the ncu-derived traffic, and the layer subsets used for profiling captures."""

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

LINE_KEYS = {"impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
             "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
             "cpu_baseline", "e2e"}


def run_bench(args, env_extra=None):
    env = dict(os.environ)
    for k in ("RANK", "LOCAL_RANK", "WORLD_SIZE"):
        env.pop(k, None)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                          capture_output=True, text=True, env=env, timeout=300)


def test_reference_arm_prints_one_contract_line():
    import bench
    res = run_bench(["--impl", "reference", "--steps", "2", "--warmup", "1",
                     "--workload", "single256_f32_r8"])
    assert res.returncode == 0, res.stderr
    lines = [l for l in res.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert LINE_KEYS <= set(line)
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["unit"] == "ZO steps/s" and line["higher_is_better"] is True
    assert line["steps"] == 2 and line["warmup"] == 1 and line["n_gpus"] == 1
    assert line["value"] > 0 and line["ms_per_step"] == pytest.approx(1e3 / line["value"])
    assert line["vs_baseline"] is None and line["dtype"] == "f64"
    cfg = line["config"]
    assert cfg["workload"] == "single256_f32_r8" and cfg["passes_per_step"] == 2 * 4 + 1
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] > 0
    assert "256 rows of matrix 0 256x256" in cb["sample"]      # rows actually sampled
    assert line["e2e"] == {"value": line["value"], "unit": "ZO steps/s",
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_forward_scheme_counts_q_plus_one_passes():
    res = run_bench(["--impl", "reference", "--steps", "1", "--warmup", "0",
                     "--workload", "single256_f32_r8", "--scheme", "forward"])
    assert res.returncode == 0, res.stderr
    line = json.loads(res.stdout.strip())
    assert line["config"]["scheme"] == "forward" and line["config"]["passes_per_step"] == 4 + 1


def test_reference_arm_runs_on_rank_zero_only():
    res = run_bench(["--impl", "reference", "--steps", "1", "--warmup", "0",
                     "--workload", "single256_f32_r8"], {"RANK": "1", "WORLD_SIZE": "2"})
    assert res.returncode == 0, res.stderr
    assert res.stdout.strip() == ""


class _ExitedProcess:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def test_clock_sampler_reads_median_clock_and_active_reasons(tmp_path):
    import bench
    rows = [
        # index, sm, max sm, power, active mask, hw_slowdown, hw_thermal, sw_thermal, sw_power_cap
        "0, 2070, 2070, 900.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 1995, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 1980, 2070, 1389.5, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, [N/A], 2070, 1.0, 0x0, Not Active, Not Active, Not Active, Not Active",   # skipped
        "garbage",
    ]
    path = tmp_path / "clocks.csv"
    path.write_text("\n".join(rows) + "\n")
    s = bench.ClockSampler(0)
    s.proc, s.path = _ExitedProcess(), str(path)
    out = s.stop()
    assert out == {"sm_mhz": 1995.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"],
                   "samples": 3}
    assert not path.exists()                     # the temporary record is removed


def test_clock_sampler_without_nvidia_smi_says_so():
    import bench
    out = bench.ClockSampler(0).stop()
    assert out["sm_mhz"] is None and out["reasons"] == ["nvidia-smi unavailable"]


def test_code_hash_ignores_comments_and_spacing(tmp_path, monkeypatch):
    import bench
    csrc = tmp_path / "paper_2608_15665_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (csrc / "k.cu").write_text("int f(int x) {\n  return x + 1;  // add one\n}\n")
    h0 = bench._code_hash(["k.cu"])
    (csrc / "k.cu").write_text("/* header */\nint f(int x) { return x + 1; }\n")
    assert bench._code_hash(["k.cu"]) == h0
    (csrc / "k.cu").write_text("int f(int x) { return x + 2; }\n")
    assert bench._code_hash(["k.cu"]) != h0


def test_layer_subsets_keep_the_shapes_and_zero_init_of_their_layers():
    import bench
    from paper_2608_15665_gb300 import workloads
    wl = workloads.get("llama7b_bf16_r32")
    assert bench.subset(wl, 0) is wl
    two = bench.subset(wl, 2)
    assert two.shapes == wl.shapes[:14] and two.r == wl.r and two.q == wl.q
    assert two.params == 2 * wl.params // 32
    lora = workloads.get("lora_opt13b_f32_r4")
    sub = bench.subset(lora, 3)
    assert sub.shapes == lora.shapes[:12]
    assert list(sub.zero_init) == [i for i in lora.zero_init if i < 12] and len(sub.zero_init) > 0
    assert bench.subset(lora, 1000).shapes == lora.shapes    # more layers than there are: all


def test_refresh_amortisation_does_not_depend_on_the_window():
    import bench
    F, K, step, ref = 25, 20, 36.0, 1.3
    # a window without a refresh and one with a refresh give the same amortised step
    w0 = K * step                               # steps 5 .. 24
    w1 = K * step + ref                         # steps 20 .. 39 (holds t = 25)
    a0 = bench.amortise_refresh(w0, K, 5, F, ref)
    a1 = bench.amortise_refresh(w1, K, 20, F, ref)
    assert a0 == pytest.approx(step + ref / F) and a1 == pytest.approx(a0)
    # two refreshes in a window of 30 steps at F = 25 (t = 25 and t = 50)
    assert bench.amortise_refresh(30 * step + 2 * ref, 30, 25, F, ref) == pytest.approx(a0)


def test_both_oracle_legs_time_the_same_sample():
    import bench
    from paper_2608_15665_gb300 import workloads
    assert bench.oracle_sample(workloads.get("llama7b_bf16_r32")) == ((0, 1024), (4, 1024))
    assert bench.oracle_sample(workloads.get("single256_f32_r8")) == ((0, 1024),)
    res = run_bench(["--impl", "reference", "--steps", "1", "--warmup", "0",
                     "--workload", "single256_f32_r8"])
    line = json.loads(res.stdout.strip())
    assert line["cpu_baseline"]["extrapolated"] is True
    assert "EXTRAPOLATED" in line["cpu_baseline"]["sample"]
    ex = line["extrapolation"]
    assert ex["weights_sampled_of"] == [256 * 256, 256 * 256] and ex["sample_seconds_per_step"] > 0


def test_single_thread_oracle_sample_runs_in_its_own_process():
    import bench
    one = bench.oracle_single_thread("single256_f32_r8", "central")
    assert one is not None and one["value"] > 0 and 0 < one["cores"] <= 1.5

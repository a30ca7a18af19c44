"""bench.py's GPU arm on a small workload: one JSON line with the keys the
measurement contract names (roofline, CPU baseline, end-to-end leg, launch
count, clocks), consistent with each other."""
import json

import pytest

import bench

pytestmark = pytest.mark.gpu


def test_gpu_arm_prints_the_contract_line(capsys, cuda_device):
    bench.main(["--workload", "tiny", "--steps", "4", "--warmup", "3", "--e2e-steps", "3",
                "--per-workload", "tiny,aq-stress"])
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["metric"] == bench.METRIC and line["unit"] == "GB/s" and line["value"] > 0
    assert line["n_gpus"] == 1 and line["steps"] == 4 and line["warmup"] == 3
    assert line["higher_is_better"] is True and line["scaling"] == "weak" and line["vs_baseline"] is None
    assert line["dtype"] == "f32" and line["data"] == "synthetic" and "tiny" in line["config"]["workload"]
    roof = line["roofline"]
    assert roof["bound"] == "hbm" and roof["unit"] == "GB/s" and roof["peak"] > 0
    assert roof["frac"] == pytest.approx(roof["achieved"] / roof["peak"], abs=1e-4)   # printed to 4 places
    assert roof["traffic"] is None or roof["traffic"] >= line["config"]["bytes_per_step"]
    cpu = line["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["value"] > 0 and cpu["cores"] >= 1 and cpu["sample"]
    e2e = line["e2e"]
    assert e2e["value"] > 0 and e2e["unit"] == "GB/s"
    assert e2e["h2d_bytes_per_step"] >= line["config"]["bytes_per_step"]   # the whole arena, padding too
    assert e2e["d2h_bytes_per_step"] > 0
    assert line["gpu_launches"] == 4                   # one step kernel per timed step
    clocks = line["clocks"]
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(clocks)
    sparsity = line["trigger_sparsity"]
    assert sparsity["steps"] > 0 and 0 <= sparsity["selected_pct"] <= 100
    assert sparsity["promotion_ratio"] == pytest.approx(sparsity["selected_pct"] / 100, abs=1e-5)
    assert 0 <= sparsity["hit_max_o_rate"] <= 1
    assert cpu["single_thread"]["cores"] == 1 and cpu["single_thread"]["value"] > 0
    per = line["per_workload"]
    assert set(per) >= {"tiny", "aq-stress", "peak_gbs"}
    for name, steps in (("tiny", 4), ("aq-stress", 4)):
        rec = per[name]
        assert rec["steps"] == steps and rec["trace_steps"][1] - rec["trace_steps"][0] + 1 == steps
        assert rec["warmup_steps"] >= 3 and rec["passes_agree"] is True
        for key in ("us_per_step", "kernel_us_mean", "kernel_us_min", "graph_us_per_step",
                    "l2_flushed_us_mean", "l2_cleaned_us_mean"):
            assert rec[key] > 0, key
        assert rec["kernel_us_min"] <= rec["kernel_us_mean"] <= rec["kernel_us_max"]
        assert rec["kernel_us_min"] <= rec["kernel_us_median"] <= rec["kernel_us_max"]
        assert rec["frac"] == pytest.approx(rec["gbs"] / per["peak_gbs"], abs=1e-3)
        assert 0 <= rec["selected_mean"] <= rec["max_o"] and rec["candidates_max"] >= 0
        assert {"sm_mhz", "reasons"} <= set(rec["clocks"])
        assert rec["trace_candidates_mean"] >= 0 and 0 <= rec["trace_selected_mean"] <= rec["max_o"]
        assert 0 <= rec["trace_hit_max_o_rate"] <= 1
    assert per["aq-stress"]["candidates_mean"] > per["aq-stress"]["max_o"]   # the contended top-k


@pytest.mark.parametrize("graph", [False, True])
def test_trace_steps_mode_times_the_trace_window(graph, capsys, cuda_device):
    """--trace-steps: the timed steps are the workload's own consecutive
    trace steps, so their candidate counts are the trace's (with --graph the
    untimed first replay's state is restored before the timed one)."""
    bench.main(["--workload", "tiny", "--trace-steps", "--steps", "6", "--warmup", "3", "--no-e2e",
                "--no-cpu-baseline", "--no-sparsity", "--no-per-workload"] + (["--graph"] if graph else []))
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    t0, t1 = line["config"]["trace_steps"]
    assert t1 - t0 + 1 == 6 and t0 >= 4 and line["config"]["arenas_cycled"] == 9
    assert line["value"] > 0 and line["gpu_launches"] == 6

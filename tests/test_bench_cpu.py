"""CPU checks of bench.py's bookkeeping: argument rules and the source hash
that keys the committed DRAM-traffic record."""
import json
import os

import pytest

import bench


def test_graph_and_flush_do_not_combine():
    with pytest.raises(SystemExit):
        bench.parse_args(["--graph", "--flush-l2"])
    assert bench.parse_args(["--graph"]).graph


def test_traffic_record_follows_the_step_kernel_sources(tmp_path, monkeypatch):
    srcs = [tmp_path / "a.cu", tmp_path / "b.cuh"]
    for i, p in enumerate(srcs):
        p.write_text(f"// source {i}\nint f{i}(int x) {{ return x + {i}; }}\n")
    prof = tmp_path / "profiles"
    prof.mkdir()
    rec = {"kernel_source_sha256_16": bench.kernel_source_hash(srcs), "traffic_bytes_per_launch": 123}
    (prof / "gnmr_step_kernel_traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic(srcs) == 123
    srcs[1].write_text("/* reworded */ // source 1, still\nint f1(int x)  {  return x + 1; }\n")
    assert bench.profiled_traffic(srcs) == 123        # comments and spacing only
    srcs[1].write_text("// source 1\nint f1(int x) { return x + 2; }\n")
    assert bench.profiled_traffic(srcs) is None


def test_committed_traffic_record_names_a_hash():
    with open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "profiles",
                           "gnmr_step_kernel_traffic.json")) as f:
        rec = json.load(f)
    assert len(rec["kernel_source_sha256_16"]) == 16 and rec["traffic_bytes_per_launch"] > 25_375_539_200


def test_exceedance_counts_only_recoverable_units_strictly_over():
    import numpy as np
    g = np.array([1.5, 2.0, 0.9, 3.0, 1.1])
    d = np.array([1.0, 1.6, 2.0, 1.5, 9.0])
    rec = np.array([1, 1, 1, 1, 0], np.uint8)
    # alpha = 1.5: units 1 and 3 (unit 0 equals it; unit 4 is not recoverable)
    # beta = 1.5: units 1 and 2 (unit 3 equals it)
    assert bench.exceedance_counts(g, d, rec, 1.5, 1.5) == (2, 2)
    assert bench.exceedance_counts(g, d, np.zeros(5, np.uint8), 1.0, 1.0) == (0, 0)


def test_reference_arm_prints_the_contract_line(capsys):
    """The reference arm (the oracle on the host cores) prints one JSON line
    with the contract's keys; its e2e moves no bytes across the host link."""
    bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "1",
                "--ref-sample-units", "8"])
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["value"] > 0 and line["unit"] == "GB/s" and line["higher_is_better"] is True
    for key in ("n_gpus", "steps", "warmup", "ms_per_step", "scaling", "vs_baseline", "dtype",
                "data", "config"):
        assert key in line, key
    assert line["vs_baseline"] is None and line["scaling"] == "weak"
    cpu = line["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] == line["value"]
    assert "units 0..7" in cpu["sample"]
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["unit"] == line["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0

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
    rec = {"records": {"tiny": {"kernel_source_sha256_16": bench.kernel_source_hash(srcs),
                                "traffic_bytes_per_launch": 123}}}
    (prof / "gnmr_step_kernel_traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic(srcs, "tiny") == 123
    assert bench.profiled_traffic(srcs, "moe") is None          # no record for that workload
    srcs[1].write_text("/* reworded */ // source 1, still\nint f1(int x)  {  return x + 1; }\n")
    assert bench.profiled_traffic(srcs, "tiny") == 123        # comments and spacing only
    srcs[1].write_text("// source 1\nint f1(int x) { return x + 2; }\n")
    assert bench.profiled_traffic(srcs, "tiny") is None


def test_committed_traffic_records_name_a_hash():
    import workloads
    with open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "profiles",
                           "gnmr_step_kernel_traffic.json")) as f:
        recs = json.load(f)["records"]
    assert "llama2-13b" in recs
    for name, rec in recs.items():
        assert name in bench.PER_WORKLOADS
        # every launch reads at least the gradient bytes once
        assert len(rec["kernel_source_sha256_16"]) == 16
        assert rec["traffic_bytes_per_launch"] >= workloads.make(name).grad_bytes


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


def test_trace_window_is_inside_the_trace_after_the_warmup():
    for T, K, W in [(20, 20, 5), (50, 20, 5), (200, 20, 5), (100, 4, 3), (3, 10, 5), (50, 1, 0)]:
        t0, k = bench.trace_window(T, K, W)
        assert k >= 1 and t0 >= 1 and t0 + k - 1 == min(T, t0 + K - 1)
        if T > W:
            assert t0 >= W + 1 and k == min(K, T - W)
    assert bench.trace_window(50, 20, 5) == (16, 20)          # centred: steps 16..35


def test_trace_steps_config_names_the_timed_trace_steps():
    """--trace-steps times consecutive trace steps after the warm-up steps,
    each with its own arena, and the config says which."""
    import workloads
    w = workloads.make("aq-stress")
    args = bench.parse_args(["--workload", "aq-stress", "--trace-steps", "--steps", "20", "--warmup", "5"])
    cfg = bench.workload_config(w, args, 0, 1)
    assert cfg["trace_steps"] == [16, 35] and cfg["arenas_cycled"] == 25
    assert bench.trace_span(w, args)[0] - args.warmup >= 1
    plain = bench.workload_config(w, bench.parse_args(["--workload", "aq-stress"]), 2, 1)
    assert "trace_steps" not in plain and plain["arenas_cycled"] == 2


def test_host_arena_follows_the_layout_and_the_trace_scales():
    """The reference arm's host-generated arena: the workload's packing,
    zeros outside the units, every unit scaled by the power of two nearest
    its trace scale (checked through the oracle's norms)."""
    import numpy as np
    import oracle
    import workloads
    w = workloads.make("tiny", shrink=8)
    step = 7
    units = np.arange(w.num_units)
    a = bench.host_arena(w, step, units, 4)
    assert a.dtype == np.float32 and a.size == w.arena_elems
    inside = np.zeros(w.arena_elems, bool)
    for o, n in zip(w.offsets, w.lengths):
        inside[o:o + n] = True
    assert np.all(a[~inside] == 0) and np.all(np.isfinite(a)) and np.all(a[inside] != 0)
    # unit s holds block[start:start+n] * 2^k: its norm is 2^k times the block slice's
    rng = np.random.default_rng([w.seed, 17, step])
    block = rng.standard_normal(bench.HOST_BLOCK, dtype=np.float32)
    block[np.abs(block) < 1e-6] = 1e-6
    norms = oracle.unit_norms(a, w.offsets, w.lengths)
    for s in (0, 5, w.num_units - 1):
        k = int(round(np.log2(w.scales[step, s])))
        start = (s * 7919) % bench.HOST_BLOCK
        ref = oracle.unit_norms(block[start:start + w.lengths[s]], [0], [w.lengths[s]])[0]
        assert norms[s] == ref * 2.0 ** k
    b = workloads.make("llama2-13b", shrink=64)
    h = bench.host_arena(b, 3, np.arange(b.num_units), 4)
    assert h.dtype == np.uint16
    bits = h[b.offsets[1]:b.offsets[1] + b.lengths[1]].astype(np.uint32) << 16
    vals = bits.view(np.float32)
    assert np.all(np.isfinite(vals)) and np.all(vals != 0)


def test_both_arms_print_the_same_config():
    """The reference arm's config object is the one the GPU arm prints for
    the same workload and arguments (the driver compares the two)."""
    import io
    import contextlib
    import workloads
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "0"])
    line = json.loads(out.getvalue().strip().splitlines()[-1])
    args = bench.parse_args(["--workload", "tiny", "--steps", "1", "--warmup", "0"])
    want = bench.workload_config(workloads.make("tiny"), args, args.arenas, 1)
    assert line["config"] == want
    assert "every step the whole 64-unit tiny layout" in line["cpu_baseline"]["sample"]
    assert "note" not in line                          # the full layout, not a sample

"""CPU-only checks of the C ABI: the library builds and loads, exports every
function that include/gnmr.h declares, its structs have the C layout, the
host-side argument checks reject bad input before any CUDA call, and the
work partition covers every unit exactly once with balanced runs."""
import ctypes
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

from paper_2606_00539_gb300 import _native as N
from paper_2606_00539_gb300 import build as native_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gnmr.h")


@pytest.fixture(scope="module")
def lib():
    native_build.build()
    return N.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gnmr_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    fns = declared_functions()
    for name in ("gnmr_create", "gnmr_step", "gnmr_destroy", "gnmr_set_thresholds",
                 "gnmr_status_string", "gnmr_last_error"):
        assert name in fns


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in N.PROTOTYPES, f"binding lacks {name}"
    assert set(N.PROTOTYPES) == set(declared_functions())


def test_struct_layout_matches_c():
    """Compile a probe against gnmr.h with gcc and compare sizeof/offsetof
    with the ctypes mirrors."""
    probe = r"""
#include <stdio.h>
#include <stddef.h>
#include "gnmr.h"
#define F(T, f) printf(#T "." #f " %zu\n", offsetof(T, f));
int main(void) {
  printf("gnmr_config %zu\n", sizeof(gnmr_config));
  printf("gnmr_stats %zu\n", sizeof(gnmr_stats));
  printf("gnmr_info %zu\n", sizeof(gnmr_info));
  F(gnmr_config, num_units) F(gnmr_config, offsets) F(gnmr_config, lengths)
  F(gnmr_config, recoverable) F(gnmr_config, dtype) F(gnmr_config, window)
  F(gnmr_config, max_o) F(gnmr_config, lock_len) F(gnmr_config, alpha_init)
  F(gnmr_config, alpha_main) F(gnmr_config, beta_init) F(gnmr_config, beta_main)
  F(gnmr_config, warmup_steps) F(gnmr_config, eps) F(gnmr_config, device)
  F(gnmr_config, num_segments) F(gnmr_config, segment_unit) F(gnmr_config, policy)
  F(gnmr_config, forced_recovery_steps) F(gnmr_config, static_warmup_steps)
  F(gnmr_config, static_fraction) F(gnmr_config, unit_cost) F(gnmr_config, loop_shape)
  F(gnmr_stats, norm) F(gnmr_stats, gnmr) F(gnmr_stats, dgnmr) F(gnmr_stats, risk)
  F(gnmr_stats, lock) F(gnmr_stats, counts) F(gnmr_stats, delta_mem)
  F(gnmr_info, num_units) F(gnmr_info, dtype) F(gnmr_info, device) F(gnmr_info, num_ctas)
  F(gnmr_info, threads_per_cta) F(gnmr_info, num_warps) F(gnmr_info, num_partials)
  F(gnmr_info, device_bytes) F(gnmr_info, arena_elems_min) F(gnmr_info, steps)
  F(gnmr_info, loop_shape) F(gnmr_info, num_runs)
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "probe.c")
        exe = os.path.join(d, "probe")
        open(src, "w").write(probe)
        subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), src, "-o", exe])
        out = subprocess.check_output([exe], text=True)
    got = dict(line.rsplit(" ", 1) for line in out.strip().splitlines())
    for cls in (N.gnmr_config, N.gnmr_stats, N.gnmr_info):
        assert int(got[cls.__name__]) == ctypes.sizeof(cls), cls.__name__
        for fname, _ in cls._fields_:
            assert int(got[f"{cls.__name__}.{fname}"]) == getattr(cls, fname).offset, fname


def test_status_strings(lib):
    for code in range(6):
        s = N.status_string(code)
        assert s.startswith("GNMR_")
    assert N.status_string(99) == "unknown gnmr_status"


def test_config_defaults(lib):
    cfg = N.gnmr_config_defaults()
    assert cfg.dtype == N.GNMR_DTYPE_BF16 and cfg.window == 8 and cfg.max_o == 4
    assert cfg.alpha_init == 1.5 and cfg.alpha_main == 1.1 and cfg.eps == 1e-8


def _valid_cfg(off, ln):
    cfg = N.gnmr_config_defaults()
    cfg.num_units = len(off)
    cfg.offsets = off.ctypes.data
    cfg.lengths = ln.ctypes.data
    return cfg


@pytest.mark.parametrize("field,value", [
    ("num_units", 0), ("dtype", 7), ("window", 0), ("max_o", -1), ("lock_len", -1),
    ("alpha_init", 0.0), ("alpha_main", float("inf")), ("beta_init", -1.0),
    ("beta_main", float("nan")), ("eps", -1e-3), ("warmup_steps", -5), ("policy", 3),
    ("forced_recovery_steps", -1), ("static_fraction", 1.5), ("static_warmup_steps", -2),
    ("loop_shape", 3), ("loop_shape", -1),
])
def test_create_rejects_bad_config_before_cuda(lib, field, value):
    off = np.array([0, 10], np.int64)
    ln = np.array([10, 5], np.int64)
    cfg = _valid_cfg(off, ln)
    setattr(cfg, field, value)
    with pytest.raises(N.GnmrError) as ei:
        N.gnmr_create(cfg)
    assert ei.value.status == N.GNMR_ERR_INVALID_ARG
    assert ei.value.detail


@pytest.mark.parametrize("offs,lens", [([-1, 0], [1, 1]), ([0, 0], [1, -2]),
                                       ([2**62, 0], [2**62, 1])])
def test_create_rejects_bad_layout(lib, offs, lens):
    off = np.array(offs, np.int64)
    ln = np.array(lens, np.int64)
    with pytest.raises(N.GnmrError) as ei:
        N.gnmr_create(_valid_cfg(off, ln))
    assert ei.value.status == N.GNMR_ERR_INVALID_ARG
    assert "unit" in ei.value.detail


def test_create_null_pointers(lib):
    cfg = N.gnmr_config_defaults()
    cfg.num_units = 3
    with pytest.raises(N.GnmrError) as ei:
        N.gnmr_create(cfg)
    assert ei.value.status == N.GNMR_ERR_INVALID_ARG
    h = ctypes.c_void_p()
    assert lib.gnmr_create(None, ctypes.byref(h)) == N.GNMR_ERR_INVALID_ARG
    assert h.value is None


def test_null_handle_calls(lib):
    assert lib.gnmr_step(None, None, 0, None, None, None) == N.GNMR_ERR_INVALID_ARG
    assert lib.gnmr_set_thresholds(None, 1.0, 1.0) == N.GNMR_ERR_INVALID_ARG
    assert lib.gnmr_get_info(None, None) == N.GNMR_ERR_INVALID_ARG
    assert lib.gnmr_destroy(None) == N.GNMR_OK


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(N, "LIB_PATH", str(tmp_path / "absent.so"))
    monkeypatch.setattr(N, "_lib", None)
    with pytest.raises(RuntimeError, match="has not been built"):
        N.load()


# ---------------------------------------------------------------------------
# Work partition (host logic of gnmr_create)
# ---------------------------------------------------------------------------

UNIT_COST = 4096
SPLIT_BYTES = 512


def _check_plan(lengths, dtype, max_warps):
    eb = 2 if dtype == N.GNMR_DTYPE_BF16 else 4
    run_unit, run_pos, first, parts = N.gnmr_plan_partition(lengths, dtype, max_warps)
    U = len(lengths)
    W = len(run_unit) - 1
    assert 1 <= W <= max_warps
    assert run_unit[0] == 0 and run_pos[0] == 0 and run_unit[-1] == U and run_pos[-1] == 0
    eff = np.maximum(lengths, 1)
    touched = [[] for _ in range(U)]
    covered = np.zeros(U, np.int64)
    costs = []
    for w in range(W):
        a = (int(run_unit[w]), int(run_pos[w]))
        b = (int(run_unit[w + 1]), int(run_pos[w + 1]))
        assert a < b, "runs must be strictly increasing (non-empty)"
        if a[1]:
            assert a[1] % (SPLIT_BYTES // eb) == 0 and a[1] < eff[a[0]]
        cost = 0
        u, p = a
        while (u, p) < b:
            stop = b[1] if u == b[0] else eff[u]
            covered[u] += stop - p
            touched[u].append(w)
            cost += (stop - p) * eb + (UNIT_COST if p == 0 else 0)
            u, p = u + 1, 0
        costs.append(cost)
    assert np.array_equal(covered, eff), "every point of every unit exactly once"
    for u in range(U):
        ws = touched[u]
        assert ws == list(range(ws[0], ws[0] + len(ws)))
        assert first[u] == ws[0] and parts[u] == len(ws)
    total = int((eff * eb + UNIT_COST).sum())
    if W > 1:
        # a run exceeds the mean by at most one split granule plus a unit's fixed cost
        assert max(costs) <= total / W + SPLIT_BYTES + UNIT_COST + eb
    return W


@pytest.mark.parametrize("seed", range(8))
def test_partition_random_layouts(lib, seed):
    rng = np.random.default_rng(seed)
    U = int(rng.integers(1, 3000))
    kind = seed % 4
    if kind == 0:
        lengths = rng.integers(0, 5000, U)
    elif kind == 1:
        lengths = np.exp(rng.uniform(0, 18, U)).astype(np.int64)
    elif kind == 2:
        lengths = np.zeros(U, np.int64)
    else:
        lengths = rng.integers(0, 3, U) * rng.integers(1, 10**7, U)
    for dtype in (N.GNMR_DTYPE_F32, N.GNMR_DTYPE_BF16):
        for max_warps in (1, 7, 4864):
            _check_plan(lengths.astype(np.int64), dtype, max_warps)


@pytest.mark.parametrize("config", [1, 2, 3, 4, 5])
def test_partition_on_workloads(lib, config):
    import workloads
    w = workloads.make(config)
    dt = N.GNMR_DTYPE_BF16 if w.dtype == "bf16" else N.GNMR_DTYPE_F32
    W = _check_plan(w.lengths, dt, 152 * 2 * 16)
    if config in (3, 4):
        assert W == 152 * 2 * 16        # big workloads use the whole grid


def _large_unit_runs(grad_bytes, num_units, grid_warps=152 * 16):
    """The run count gnmr_create plans for the large-unit loop: about 16 runs
    per warp of 64-256 KiB of cost each, never fewer than one per warp."""
    cost = grad_bytes + UNIT_COST * num_units
    run = min(max(cost // (grid_warps * 16), 64 << 10), 256 << 10)
    return max(grid_warps, -(-cost // run)), run


@pytest.mark.parametrize("config", [2, 3, 4])
def test_partition_of_dynamic_runs(lib, config):
    """The many-runs plans of the large-unit loop (37K-121K runs): the same
    invariants, and every run within a granule and a unit's fixed cost of
    the run size."""
    import workloads
    w = workloads.make(config)
    dt = N.GNMR_DTYPE_BF16 if w.dtype == "bf16" else N.GNMR_DTYPE_F32
    R, run = _large_unit_runs(w.grad_bytes, w.num_units)
    assert R > 8 * 152 * 16
    W = _check_plan(w.lengths, dt, int(R))
    assert R - 1 <= W <= R


def test_partition_rejects_bad_input(lib):
    with pytest.raises(N.GnmrError):
        N.gnmr_plan_partition(np.array([5, -1], np.int64), N.GNMR_DTYPE_F32, 4)
    with pytest.raises(N.GnmrError):
        N.gnmr_plan_partition(np.array([5], np.int64), 9, 4)


def test_monitor_rejects_unknown_loop_shape(lib):
    from paper_2606_00539_gb300 import Monitor
    with pytest.raises(ValueError, match="loop_shape"):
        Monitor(np.array([0], np.int64), np.array([4], np.int64), loop_shape="medium")

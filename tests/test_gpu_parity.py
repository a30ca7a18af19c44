"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Masks, locks and counts must match exactly; norms, GNMR, Delta-GNMR and R to
a relative 1e-5.  The workloads run in lockstep with the oracle (see
trace_driver) so that every rounded decision has margin."""
import math
from types import SimpleNamespace

import numpy as np
import pytest

import oracle
import workloads
from paper_2606_00539_gb300 import Monitor
from paper_2606_00539_gb300 import _native as N
from tests import trace_driver as TD
from tests.golden import hand_traces

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def _monitor(w, **over):
    kw = w.monitor_kwargs()
    kw.update(over)
    return Monitor(w.offsets, w.lengths, device=0, **kw)


def _policy_kwargs(cfg):
    from fractions import Fraction
    return dict(policy=int(cfg.get("policy", 0)), forced_recovery_steps=int(cfg.get("forced", 0)),
                static_warmup_steps=int(cfg.get("static_warmup", 0)),
                static_fraction=float(cfg.get("static_fraction", Fraction(1, 4))))


def _run_lockstep(w, steps=None, every=1):
    tr = TD.LockstepTrace(w, "cuda:0", _monitor)
    try:
        for t in range(steps or w.steps):
            norms, res, got = tr.step(t)
            if t % every == 0 or t == (steps or w.steps) - 1:
                TD.compare(norms, res, got, RTOL)
    finally:
        tr.close()
    return tr


# ---------------------------------------------------------------------------
# The five workloads (small cases: several tiles per unit and ragged tails)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("config,shrink,steps", [
    ("tiny", 1, None),           # 64 fp32 units, 200 steps
    ("llama2-1.3b", 8, 60),      # 168 bf16 units, dims / 8
    ("llama2-13b", 16, None),    # 280 bf16 units, dims / 16, 20 steps
    ("moe", 16, 30),             # 5454 bf16 units with unrouted experts
    ("aq-stress", 1, 20),        # 100K fp32 units, contended top-64
])
def test_workload_parity(config, shrink, steps, cuda_device):
    w = workloads.make(config, shrink=shrink, steps=steps)
    tr = _run_lockstep(w)
    assert sum(r.attempts for r in tr.records) < 10 * w.steps


@pytest.mark.parametrize("config,group,shrink,steps", [
    ("llama2-13b", "block", 16, None),     # 40 layer units of 7 tensors each
    ("llama2-1.3b", "block", 8, 40),
    ("moe", "expert", 16, 20),             # attention + each expert as one unit
    ("moe", "block", 32, 20),
])
def test_block_level_units_parity(config, group, shrink, steps, cuda_device):
    """Units spanning several tensors (Sec. 3.4): the unit norm covers all of
    its tensors and the whole block shares one decision."""
    w = workloads.make(config, shrink=shrink, steps=steps, group=group)
    assert w.num_units < w.num_segments
    _run_lockstep(w)


def _large_shape_monitor(w, **over):
    return _monitor(w, loop_shape="large", **over)


@pytest.mark.parametrize("config,group,shrink,steps", [
    ("tiny", "tensor", 1, 60),
    ("llama2-13b", "tensor", 16, None),
    ("aq-stress", "tensor", 1, 10),
    ("moe", "expert", 16, 12),
])
def test_large_unit_loop_shape_parity(config, group, shrink, steps, cuda_device):
    """The large-unit loop shape (twice the loads in flight per warp, half
    the resident warps) forced on the small cases, which would otherwise run
    the small-unit shape: same bar against the oracle."""
    w = workloads.make(config, shrink=shrink, steps=steps, group=group)
    tr = TD.LockstepTrace(w, "cuda:0", _large_shape_monitor)
    try:
        assert tr.mon.info()["loop_shape"] == N.GNMR_LOOP_LARGE_UNITS
        for t in range(w.steps):
            norms, res, got = tr.step(t)
            TD.compare(norms, res, got, RTOL)
    finally:
        tr.close()


def test_loop_shape_follows_the_mean_unit_size(cuda_device):
    """GNMR_LOOP_AUTO takes the large-unit shape at >= 1 MiB per unit."""
    for config, want in (("tiny", N.GNMR_LOOP_SMALL_UNITS), ("aq-stress", N.GNMR_LOOP_SMALL_UNITS),
                         ("llama2-1.3b", N.GNMR_LOOP_LARGE_UNITS), ("llama2-13b", N.GNMR_LOOP_LARGE_UNITS),
                         ("moe", N.GNMR_LOOP_LARGE_UNITS)):
        w = workloads.make(config)
        with _monitor(w) as mon:
            assert mon.info()["loop_shape"] == want, config
        for shape, code in (("small", N.GNMR_LOOP_SMALL_UNITS), ("large", N.GNMR_LOOP_LARGE_UNITS)):
            with _monitor(w, loop_shape=shape) as mon:
                assert mon.info()["loop_shape"] == code


def test_large_unit_loop_takes_runs_dynamically(cuda_device):
    """The large-unit loop plans about 16 runs per warp (64-256 KiB each), and
    the small-unit loop one run per warp."""
    for config in ("llama2-1.3b", "llama2-13b", "moe", "tiny", "aq-stress"):
        w = workloads.make(config)
        with _monitor(w) as mon:
            info = mon.info()
            cost = w.grad_bytes + 4096 * w.num_units
            if info["loop_shape"] == N.GNMR_LOOP_LARGE_UNITS:
                assert info["num_runs"] > 4 * info["num_warps"], config
                assert (64 << 10) * 0.99 <= cost / info["num_runs"] <= (256 << 10) * 1.01, config
                assert info["num_partials"] >= info["num_runs"]
            else:
                assert info["num_runs"] == info["num_warps"], config
            assert info["num_ctas"] * info["threads_per_cta"] // 32 >= info["num_warps"]


def test_two_handles_stepping_concurrently_do_not_interfere(cuda_device):
    """Two handles of the same large-unit layout (dynamic runs: each handle
    has its own run counter) stepping on two streams at once, with no host
    synchronisation between them, give bit-identical outputs to a third
    handle stepping alone."""
    import torch
    w = workloads.make("llama2-1.3b", shrink=2, steps=6)
    filler = workloads.Filler(w, cuda_device)
    arenas = []
    for t in range(w.steps):
        a = filler.new_arena()
        filler.fill(a, t)
        arenas.append(a)
    torch.cuda.synchronize()
    mons = [_monitor(w) for _ in range(3)]
    try:
        assert mons[0].info()["num_runs"] > mons[0].info()["num_warps"]
        streams = [torch.cuda.Stream(cuda_device) for _ in range(2)]
        stats = [m.new_stats() for m in mons]
        masks = [torch.empty(w.num_units, dtype=torch.uint8, device=cuda_device) for _ in mons]
        history = [[] for _ in mons]
        for t in range(w.steps):
            for k in range(2):                                   # concurrent, no sync between
                mons[k].step(arenas[t], mask=masks[k], stats=stats[k], stream=streams[k])
            torch.cuda.synchronize()
            mons[2].step(arenas[t], mask=masks[2], stats=stats[2])   # alone
            torch.cuda.synchronize()
            for k in range(3):
                history[k].append({n: v.clone() for n, v in stats[k].items()} | {"mask": masks[k].clone()})
        for t in range(w.steps):
            for k in range(2):
                for name, v in history[2][t].items():
                    assert torch.equal(history[k][t][name], v), (t, k, name)
    finally:
        for m in mons:
            m.close()


def test_segments_in_any_order_and_units_without_segments(cuda_device):
    import torch
    rng = np.random.default_rng(21)
    n = 400_000
    off = np.array([5000, 0, 123_457, 300_001, 77, 200_000, 350_000], np.int64)
    ln = np.array([100_000, 77, 3, 99_999, 4_923, 0, 50_000], np.int64)
    unit = np.array([3, 0, 3, 1, 0, 1, 4], np.int32)                # unit 2 has no segment
    U = 5
    base = _random_arena(rng, n, "bf16").to(cuda_device)
    mon = Monitor(off, ln, dtype="bf16", segment_unit=unit, num_units=U, window=2, max_o=2,
                  lock_len=1, device=0)
    ctl = oracle.Controller(U, window=2, max_o=2, lock_len=1, alpha=(1.5, 1.1), beta=(1.5, 1.5))
    stats = mon.new_stats()
    try:
        for t in range(4):
            dev = (base.float() * float(1.0 + 0.37 * t)).to(torch.bfloat16)
            norms = oracle.unit_norms_segmented(_host_view(dev), off, ln, unit, U)
            assert norms[2] == 0.0
            res = ctl.step(norms)
            mask = mon.step(dev, stats=stats)
            got = {k: v.cpu().numpy() for k, v in stats.items()}
            got["mask"] = mask.cpu().numpy()
            np.testing.assert_allclose(got["norm"], norms, rtol=RTOL, atol=0)
            np.testing.assert_allclose(got["gnmr"], res.gnmr, rtol=RTOL, atol=0)
    finally:
        mon.close()
        ctl.close()


@pytest.mark.parametrize("seed", [1, 2])
def test_tiny_more_seeds(seed, cuda_device):
    _run_lockstep(workloads.make("tiny", seed=seed, steps=120))


# ---------------------------------------------------------------------------
# Hand-derived traces replayed on the GPU (exact norms: one fp32 element each)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("trace", hand_traces.all_traces(), ids=lambda t: t.name)
def test_hand_trace_on_gpu(trace, cuda_device):
    import torch
    cfg = trace.cfg
    U = int(cfg["units"])
    off = np.arange(U, dtype=np.int64) * 4            # one element per unit, 16 B apart
    ln = np.ones(U, np.int64)
    mon = Monitor(off, ln, dtype="f32", recoverable=[int(x) for x in cfg["recoverable"]],
                  window=int(cfg["window"]), max_o=int(cfg["max_o"]),
                  lock_len=int(cfg["lock_len"]),
                  alpha=(float(cfg["alpha_init"]), float(cfg["alpha_main"])),
                  beta=(float(cfg["beta_init"]), float(cfg["beta_main"])),
                  warmup_steps=int(cfg["warmup"]), eps=float(cfg["eps"]), device=0,
                  **_policy_kwargs(cfg))
    stats = mon.new_stats()
    arena = torch.zeros(4 * U, dtype=torch.float32, device=cuda_device)
    try:
        for st in trace.steps:
            arena[off] = torch.tensor([float(x) for x in st.n], dtype=torch.float32,
                                      device=cuda_device)
            mask = mon.step(arena, stats=stats).cpu().numpy()
            g = {k: v.cpu().numpy() for k, v in stats.items()}
            for b in range(U):
                for key, want in (("gnmr", st.gnmr[b]), ("dgnmr", st.dgnmr[b]),
                                  ("risk", st.risk[b])):
                    want = float(want)
                    if math.isinf(want):
                        assert g[key][b] == want, (st.t, b, key)
                    else:
                        assert g[key][b] == pytest.approx(want, rel=1e-6, abs=1e-12), (st.t, b, key)
            assert list(np.nonzero(mask)[0]) == st.selected, st.t
            assert list(g["lock"]) == st.lock_after, st.t
            assert list(g["counts"]) == [len(st.candidates), len(st.selected)], st.t
    finally:
        mon.close()


# ---------------------------------------------------------------------------
# Edge cases
# ---------------------------------------------------------------------------

def _random_arena(rng, n, dtype, scale=1.0):
    import torch
    x = torch.from_numpy((rng.standard_normal(n) * scale).astype(np.float32))
    return x.to(torch.bfloat16) if dtype == "bf16" else x


def _host_view(t):
    import torch
    t = t.cpu()
    return t.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else t.numpy()


def _parity_on_norms(off, ln, dev_arena, make_step, mon_kw, ctl_kw, steps, recoverable=None):
    """Runs `steps` steps.  make_step(t, attempt, bad) writes step t's
    gradients into dev_arena; when the oracle finds a decision without margin
    it is called again with attempt + 1 and the units to redraw (the oracle
    state is rolled back first).  Every output is compared with the oracle."""
    U = len(off)
    rec = np.ones(U, np.uint8) if recoverable is None else np.asarray(recoverable, np.uint8)
    mon = Monitor(off, ln, device=0, recoverable=rec, **mon_kw)
    ctl = oracle.Controller(U, recoverable=rec, **ctl_kw)
    stats = mon.new_stats()
    margin_cfg = SimpleNamespace(recoverable=rec, warmup_steps=0,
                                 **{k: ctl_kw[k] for k in ("alpha", "beta", "window", "max_o")})
    try:
        for t in range(steps):
            attempt, bad = 0, []
            while True:
                make_step(t, attempt, bad)
                norms = oracle.unit_norms(_host_view(dev_arena), off, ln)
                before = ctl.get_state()
                res = ctl.step(norms)
                bad = TD.margin_violations(before, res, margin_cfg, t + 1)
                if not bad:
                    break
                ctl.set_state(before)
                attempt += 1
                assert attempt < 30, f"no decision margin at step {t + 1}: units {bad[:8]}"
            mask = mon.step(dev_arena, stats=stats)
            got = {k: v.cpu().numpy() for k, v in stats.items()}
            got["mask"] = mask.cpu().numpy()
            TD.compare(norms, res, got, RTOL)
    finally:
        mon.close()
        ctl.close()


@pytest.mark.parametrize("shape", ["small", "large"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_unaligned_overlapping_and_empty_units(dtype, shape, cuda_device):
    """Units at odd element offsets, overlapping units, gaps, zero-length and
    one-element units, and a unit spanning many warps."""
    import torch
    rng = np.random.default_rng(11)
    n = 3_000_001
    off = np.array([0, 1, 3, 7, 100, 101, 5, 2_000_000, 17, 999_999, 0, 2_999_990], np.int64)
    ln = np.array([1, 2, 13, 0, 1, 777, 2_000_000, 1_000_001, 0, 3, 3_000_001, 11], np.int64)
    base = _random_arena(rng, n, "f32").to(cuda_device)
    dev = torch.empty(n, dtype=torch.bfloat16 if dtype == "bf16" else torch.float32,
                      device=cuda_device)
    gen = torch.Generator(device=cuda_device)

    def make_step(t, attempt, bad):
        # fresh elementwise noise per step (and per attempt): every unit's
        # norm moves on its own
        gen.manual_seed(1000 * t + attempt)
        noise = torch.randn(n, generator=gen, device=cuda_device)
        x = base * (1.0 + 0.3 * noise)
        if t == 3:
            x[2_000_000:2_000_500] *= 40.0
        dev.copy_(x.to(dev.dtype))

    _parity_on_norms(off, ln, dev, make_step,
                     dict(dtype=dtype, window=2, max_o=3, lock_len=2, alpha=1.2, beta=1.2,
                          loop_shape=shape),
                     dict(window=2, max_o=3, lock_len=2, alpha=(1.2, 1.2), beta=(1.2, 1.2)), 6)


def test_dynamic_runs_with_unaligned_special_and_empty_units(cuda_device):
    """The large-unit loop with many more runs than warps (a 400 MB bf16 arena,
    ~6,000 runs of 64 KiB): units at odd offsets, overlapping units, empty and
    one-element units, a unit over the whole arena, a unit that turns NaN and
    one whose squares overflow fp32 (the exact path) at some steps."""
    import torch
    n = 200_000_003
    rng = np.random.default_rng(31)
    off = [0, 1, 3, 7, 11, 150_000_001, 5, 0, 99_999_999, 123]
    ln = [1, 0, 40_000_001, 13, 60_000_000, 49_999_999, 20_000_003, n, 2, 3_000_000]
    for _ in range(30):                                   # assorted units in [0, 100M), some overlapping
        o = int(rng.integers(0, 88_000_000))
        off.append(o)
        ln.append(int(rng.integers(100_000, 12_000_000)))
    off = np.array(off, np.int64)
    ln = np.array(ln, np.int64)
    gen = torch.Generator(device=cuda_device)
    gen.manual_seed(5)
    base = torch.randn(n, generator=gen, device=cuda_device)
    dev = torch.empty(n, dtype=torch.bfloat16, device=cuda_device)

    def make_step(t, attempt, bad):
        gen.manual_seed(7000 + 100 * t + attempt)
        noise = torch.randn(n, generator=gen, device=cuda_device)
        x = base * (1.0 + 0.3 * noise)
        if t == 2:
            x[199_999_990] = float("nan")                     # units 5 and 7 only
        if t == 4:
            x[11 + 1_000:11 + 2_000] = 3e25                    # unit 4: fp32 squares overflow
        dev.copy_(x.to(torch.bfloat16))

    mon_kw = dict(dtype="bf16", window=3, max_o=4, lock_len=2, alpha=1.2, beta=1.2, loop_shape="large")
    with Monitor(off, ln, device=0, **mon_kw) as mon:
        info = mon.info()
        assert info["loop_shape"] == N.GNMR_LOOP_LARGE_UNITS
        assert info["num_runs"] > 2 * info["num_warps"]
    _parity_on_norms(off, ln, dev, make_step, mon_kw,
                     dict(window=3, max_o=4, lock_len=2, alpha=(1.2, 1.2), beta=(1.2, 1.2)), 7)


def _per_unit_levels_arena(rng, ln, steps, sigma, device, zero_units=()):
    """Packed fp32 units; step t of unit u is base * level[t, u].  Returns
    (offsets, arena, make_step) with per-unit margin repair."""
    import torch
    off = np.concatenate([[0], np.cumsum(ln)[:-1]]).astype(np.int64)
    base = _random_arena(rng, int(ln.sum()), "f32").to(device)
    unit_of = torch.from_numpy(np.repeat(np.arange(len(ln)), ln)).to(device)
    levels = np.exp(sigma * rng.standard_normal((steps, len(ln))))
    for u in zero_units:
        levels[:, u] = 0.0
    dev = base.clone()
    cur = {}

    def make_step(t, attempt, bad):
        if attempt == 0:
            cur["lv"] = levels[t].copy()
        for u in bad:
            cur["lv"][u] *= math.exp(rng.uniform(-0.01, 0.01))
        lv = torch.from_numpy(cur["lv"].astype(np.float32)).to(device)
        dev.copy_(base * lv[unit_of])

    return off, dev, make_step


def test_nonfinite_gradients(cuda_device):
    """NaN/Inf in a unit: R = +inf (selected first, ties by index), and the
    unit's A, Q, k stay as they were -- checked over the following steps."""
    rng = np.random.default_rng(13)
    U, L = 16, 4096
    ln = np.full(U, L, np.int64)
    off, dev, base_step = _per_unit_levels_arena(rng, ln, 9, 0.2, cuda_device)

    def make_step(t, attempt, bad):
        base_step(t, attempt, bad)
        if t == 4:
            dev[5 * L + 17] = float("nan")
            dev[9 * L + 3] = float("inf")
            dev[2 * L + 100] = float("-inf")

    _parity_on_norms(off, ln, dev, make_step,
                     dict(dtype="f32", window=3, max_o=2, lock_len=1, alpha=1.5, beta=1.5),
                     dict(window=3, max_o=2, lock_len=1, alpha=(1.5, 1.5), beta=(1.5, 1.5)), 9)


@pytest.mark.parametrize("window", [1, 9, 13, 24])
def test_window_lengths(window, cuda_device):
    """Delta-GNMR windows outside the standard 5 and 8: a single entry, and
    windows longer than the eight entries the epilogue reads per batch (the
    ring wraps mid-batch and leaves a remainder); enough steps that every
    window fills and wraps."""
    rng = np.random.default_rng(100 + window)
    U = 300
    ln = rng.integers(1, 2000, U).astype(np.int64)
    steps = window + 7
    off, dev, make_step = _per_unit_levels_arena(rng, ln, steps, 0.3, cuda_device)
    _parity_on_norms(off, ln, dev, make_step,
                     dict(dtype="f32", window=window, max_o=6, lock_len=2, alpha=1.3, beta=1.2),
                     dict(window=window, max_o=6, lock_len=2, alpha=(1.3, 1.3), beta=(1.2, 1.2)), steps)


@pytest.mark.parametrize("max_o,lock_len,thr", [(0, 3, 1.05), (10_000, 0, 1.05), (7, 2, 0.9)])
def test_budget_extremes_and_ties(max_o, lock_len, thr, cuda_device):
    """maxO = 0 (never select), maxO >= U (plain threshold), and thresholds
    below 1 so that every unit ties at t = 1 (index order decides); some units
    are not recoverable and some are all zeros."""
    rng = np.random.default_rng(14)
    U = 5000
    ln = rng.integers(1, 300, U).astype(np.int64)
    rec = (rng.random(U) < 0.9).astype(np.uint8)
    off, dev, make_step = _per_unit_levels_arena(rng, ln, 8, 0.5, cuda_device,
                                                 zero_units=range(0, U, 97))
    _parity_on_norms(off, ln, dev, make_step,
                     dict(dtype="f32", window=2, max_o=max_o, lock_len=lock_len, alpha=thr, beta=thr),
                     dict(window=2, max_o=max_o, lock_len=lock_len, alpha=(thr, thr), beta=(thr, thr)),
                     8, recoverable=rec)


@pytest.mark.parametrize("shape", ["small", "large"])
def test_tiny_and_huge_fp32_values_take_the_exact_path(shape, cuda_device):
    """fp32 squares underflow below ~1e-19 and overflow above ~1.8e19; the
    kernel's fp64 fallback keeps the norm within rounding of the oracle."""
    import torch
    rng = np.random.default_rng(12)
    parts = [rng.standard_normal(5000) * 1e-30, rng.standard_normal(5000) * 1e25,
             rng.standard_normal(5000), np.concatenate([np.full(10, 1e-44), np.zeros(90)]),
             rng.standard_normal(70000) * 3e-21]
    host = np.concatenate(parts).astype(np.float32)
    off = np.cumsum([0] + [len(p) for p in parts[:-1]]).astype(np.int64)
    ln = np.array([len(p) for p in parts], np.int64)
    dev = torch.from_numpy(host).to(cuda_device)
    mon = Monitor(off, ln, dtype="f32", device=0, loop_shape=shape)
    stats = mon.new_stats()
    try:
        mon.step(dev, stats=stats)
        got = stats["norm"].cpu().numpy()
    finally:
        mon.close()
    want = oracle.unit_norms(host, off, ln)
    assert np.all(want > 0)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=0)


def test_all_units_tie_under_contention(cuda_device):
    """100K units, thresholds 0.5: at t = 1 every unit has R = 2; the top-64
    must be units 0..63."""
    import torch
    U = 100_000
    off = np.arange(U, dtype=np.int64) * 4
    ln = np.full(U, 4, np.int64)
    dev = torch.ones(4 * U, dtype=torch.float32, device=cuda_device)
    mon = Monitor(off, ln, dtype="f32", max_o=64, lock_len=3, alpha=0.5, beta=0.5, window=4, device=0)
    stats = mon.new_stats()
    try:
        mask = mon.step(dev, stats=stats).cpu().numpy()
        assert list(np.nonzero(mask)[0]) == list(range(64))
        assert list(stats["counts"].cpu().numpy()) == [U, 64]
        assert np.all(stats["risk"].cpu().numpy() == 2.0)
    finally:
        mon.close()


def test_threshold_override_and_schedule(cuda_device):
    """gnmr_set_thresholds overrides alpha_t/beta_t until reset with NaN."""
    w = workloads.make("tiny", seed=5, steps=40, shrink=8)
    tr = TD.LockstepTrace(w, "cuda:0", _monitor)
    try:
        for t in range(w.steps):
            if t == 20:
                tr.mon.set_thresholds(1.05, 1.2)
            if t == 30:
                tr.mon.set_thresholds(float("nan"), float("nan"))
            a, b = (1.05, 1.2) if 20 <= t < 30 else (math.nan, math.nan)
            norms, res, got = tr.step(t, a, b)
            TD.compare(norms, res, got, RTOL)
    finally:
        tr.close()


@pytest.mark.parametrize("config,shrink", [("llama2-13b", 32), ("tiny", 1), ("moe", 32)])
def test_pinned_host_arena_is_read_in_place(config, shrink, cuda_device):
    """gnmr_step on a pinned host arena (read in place over the host link)
    gives bitwise the outputs of the same arena in device memory, and so do
    the partial sums; an unpinned host tensor is refused."""
    import torch
    w = workloads.make(config, shrink=shrink, steps=4)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    host = torch.empty(arena.numel(), dtype=arena.dtype, pin_memory=True)
    m_dev, m_host = _monitor(w), _monitor(w)
    s_dev, s_host = m_dev.new_stats(), m_host.new_stats()

    def bits(x):
        return x.view(torch.int64) if x.dtype == torch.float64 else x

    try:
        for t in range(w.steps):
            f.fill(arena, t)
            host.copy_(arena)
            a = m_dev.step(arena, stats=s_dev)
            b = m_host.step(host, stats=s_host)
            torch.cuda.synchronize()
            assert torch.equal(a, b), f"mask, step {t + 1}"
            for k in s_dev:
                assert torch.equal(bits(s_dev[k]), bits(s_host[k])), f"{k}, step {t + 1}"
        assert torch.equal(bits(m_dev.step_partials(arena)), bits(m_host.step_partials(host)))
        with pytest.raises(ValueError, match="pinned"):
            m_host.step(torch.zeros(8, dtype=arena.dtype))
    finally:
        m_dev.close()
        m_host.close()


def test_prepared_step_matches_step(cuda_device):
    """Monitor.prepare_step: the prepared call gives bitwise the outputs of
    step() on the same arena contents, follows new contents written into the
    same storage, and refuses to run after close()."""
    import torch
    w = workloads.make("aq-stress", shrink=4, steps=5)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    m_a, m_b = _monitor(w), _monitor(w)
    s_a, s_b = m_a.new_stats(), m_b.new_stats()
    mask_b = torch.empty(w.num_units, dtype=torch.uint8, device=cuda_device)
    run = m_b.prepare_step(arena, mask=mask_b, stats=s_b)
    try:
        for t in range(w.steps):
            f.fill(arena, t)
            a = m_a.step(arena, stats=s_a)
            b = run()
            torch.cuda.synchronize()
            assert b is mask_b and torch.equal(a, b), f"mask, step {t + 1}"
            for k in s_a:
                x, y = s_a[k], s_b[k]
                if x.dtype == torch.float64:
                    x, y = x.view(torch.int64), y.view(torch.int64)
                assert torch.equal(x, y), f"{k}, step {t + 1}"
    finally:
        m_a.close()
        m_b.close()
    with pytest.raises(ValueError, match="closed"):
        run()


@pytest.mark.parametrize("shape", ["small", "large"])
def test_deterministic_across_handles_and_runs(shape, cuda_device):
    import torch
    w = workloads.make("llama2-13b", shrink=32, steps=4)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    outs = []
    for _ in range(2):
        mon = _monitor(w, loop_shape=shape)
        stats = mon.new_stats()
        vals = []
        for t in range(w.steps):
            f.fill(arena, t)
            mon.step(arena, stats=stats)
            vals.append(stats["norm"].cpu().numpy().copy())
        mon.close()
        outs.append(np.stack(vals))
    assert np.array_equal(outs[0].view(np.uint64), outs[1].view(np.uint64))


def test_errors_leave_state_unchanged(cuda_device):
    import torch
    rng = np.random.default_rng(15)
    U, L = 8, 1000
    off = np.arange(U, dtype=np.int64) * L
    ln = np.full(U, L, np.int64)
    dev = _random_arena(rng, U * L, "bf16").to(cuda_device)
    mon = Monitor(off, ln, dtype="bf16", device=0)
    ctl = oracle.Controller(U, window=8, max_o=4, lock_len=1, alpha=(1.5, 1.1), beta=(1.5, 1.5))
    stats = mon.new_stats()
    mask = torch.empty(U, dtype=torch.uint8, device=cuda_device)
    try:
        h = mon._h
        # arena shorter than the layout
        with pytest.raises(N.GnmrError) as ei:
            N.gnmr_step(h, dev.data_ptr(), U * L - 1, 0, mask.data_ptr(), None)
        assert ei.value.status == N.GNMR_ERR_LAYOUT
        # misaligned arena pointer (odd byte address for bf16)
        with pytest.raises(N.GnmrError) as ei:
            N.gnmr_step(h, dev.data_ptr() + 1, U * L, 0, mask.data_ptr(), None)
        assert ei.value.status == N.GNMR_ERR_INVALID_ARG
        with pytest.raises(N.GnmrError) as ei:
            N.gnmr_step(h, dev.data_ptr(), U * L, 0, None, None)
        assert ei.value.status == N.GNMR_ERR_INVALID_ARG
        with pytest.raises(N.GnmrError):
            mon.set_thresholds(-1.0, 1.0)
        assert mon.info()["steps"] == 0
        for t in range(3):
            dev.mul_(1.0 + t)
            norms = oracle.unit_norms(_host_view(dev), off, ln)
            res = ctl.step(norms)
            m = mon.step(dev, stats=stats)
            got = {k: v.cpu().numpy() for k, v in stats.items()}
            got["mask"] = m.cpu().numpy()
            TD.compare(norms, res, got, RTOL)
        assert mon.info()["steps"] == 3
    finally:
        mon.close()
        ctl.close()


def test_mask_only_and_side_stream(cuda_device):
    import torch
    w = workloads.make("tiny", seed=7, steps=12, shrink=4)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    a = _monitor(w)
    b = _monitor(w)
    stats = b.new_stats()
    side = torch.cuda.Stream(cuda_device)
    try:
        for t in range(w.steps):
            f.fill(arena, t)
            torch.cuda.synchronize()
            with torch.cuda.stream(side):
                m1 = a.step(arena, stream=side)
            m2 = b.step(arena, stats=stats)
            side.synchronize()
            torch.cuda.synchronize()
            assert torch.equal(m1, m2)
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("config,shrink,steps", [("tiny", 4, 30),
                                                 ("llama2-1.3b", 2, 10)])   # dynamic runs
def test_cuda_graph_replay_advances_steps(config, shrink, steps, cuda_device):
    """The step is one launch with no host synchronisation: captured once in a
    CUDA graph and replayed, it matches the oracle step by step (the step
    counter, the thresholds and the large-unit loop's run counter live on the
    device and are reset by the kernel)."""
    import torch
    w = workloads.make(config, seed=9, steps=steps, shrink=shrink)
    tr = TD.LockstepTrace(w, "cuda:0", _monitor)
    mask = torch.empty(w.num_units, dtype=torch.uint8, device=cuda_device)
    s = torch.cuda.Stream(cuda_device)
    g = torch.cuda.CUDAGraph()
    try:
        with torch.cuda.graph(g, stream=s):
            tr.mon.step(tr.arena, mask=mask, stats=tr.stats, stream=s)
        # capturing does not run the kernel: the device state is still at t = 0

        def replay():
            g.replay()
            return mask

        for t in range(w.steps):
            norms, res, got = tr.step(t, gpu_step=replay)
            TD.compare(norms, res, got, RTOL)
    finally:
        tr.close()


@pytest.mark.parametrize("config,shrink", [("aq-stress", 8), ("llama2-13b", 16)])
def test_steps_wait_for_the_kernel_that_writes_the_arena(config, shrink, cuda_device):
    """Steps enqueued right behind the kernel that writes their arena, with no
    host synchronisation in between: fill, step, fill, step, ... on one
    stream.  Each step must see its own step's gradients (its norms equal the
    oracle's on that step's bytes, regenerated separately afterwards), so a
    step never starts reading before the writer has finished."""
    import torch
    import oracle
    w = workloads.make(config, shrink=shrink, steps=6)
    filler = workloads.Filler(w, cuda_device)
    arena = filler.new_arena()
    mon = _monitor(w)
    norms = torch.empty((w.steps, w.num_units), dtype=torch.float64, device=cuda_device)
    stats = mon.new_stats()
    try:
        torch.cuda.synchronize()
        for t in range(w.steps):
            filler.fill(arena, t)                    # torch's current stream, then the step on it
            mon.step(arena, stats=dict(stats, norm=norms[t]))
        torch.cuda.synchronize()
        got = norms.cpu().numpy()
        check = filler.new_arena()
        for t in range(w.steps):
            filler.fill(check, t)
            host = check.cpu()
            view = host.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16" else host.numpy()
            want = oracle.unit_norms_threaded(view, w.offsets, w.lengths, 8)
            np.testing.assert_allclose(got[t], want, rtol=RTOL, atol=0, err_msg=f"step {t + 1}")
    finally:
        mon.close()

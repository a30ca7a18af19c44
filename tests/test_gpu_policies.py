"""Policy variants on the GPU against the oracle: the admission cap (the
Remark on the maxO budget), the forced high-fidelity warm-up (App. E.7), the
ADAPT-style static top fraction (App. E.4), and the Delta M_t statistic
(Eq. generic-memory-bound)."""
import math

import numpy as np
import pytest

import workloads
from paper_2606_00539_gb300 import Monitor
from tests import trace_driver as TD

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def _monitor(w, **over):
    kw = w.monitor_kwargs()
    kw.update(over)
    return Monitor(w.offsets, w.lengths, device=0, **kw)


def _run(w, policy, steps=None, check=None):
    tr = TD.LockstepTrace(w, "cuda:0", _monitor, policy=policy)
    try:
        for t in range(steps or w.steps):
            norms, res, got = tr.step(t)
            TD.compare(norms, res, got, RTOL)
            if check:
                check(t + 1, tr, res, got)
    finally:
        tr.close()
    return tr


@pytest.mark.parametrize("config,shrink,steps", [("tiny", 2, 80), ("aq-stress", 4, 20),
                                                 ("llama2-13b", 32, None),
                                                 ("llama2-1.3b", 2, 30)])   # dynamic runs
def test_admission_cap_parity(config, shrink, steps, cuda_device):
    w = workloads.make(config, shrink=shrink, steps=steps)
    seen = {"over": False}

    def check(t, tr, res, got):
        seen["over"] |= res.n_selected > w.max_o          # |A_t| may exceed maxO here

    _run(w, dict(policy=1), check=check)
    if config == "aq-stress":
        assert seen["over"]


def test_forced_warmup_parity(cuda_device):
    w = workloads.make("moe", shrink=32, steps=20)

    def check(t, tr, res, got):
        if t <= 4:
            assert np.array_equal(got["mask"], w.recoverable) and got["counts"][0] == 0

    _run(w, dict(forced_recovery_steps=4), check=check)


@pytest.mark.parametrize("policy", [dict(policy=1, forced_recovery_steps=1),
                                    dict(policy=2, static_warmup_steps=1, static_fraction=0.1),
                                    dict(policy=2, static_warmup_steps=0, static_fraction=0.1)])
def test_short_warmups_parity(policy, cuda_device):
    """One-step (and, for the static policy, empty) warm-ups: the all-on
    step is the first step, and the static choice rests on one step's GNMR
    (or on none: every sum 0, the lowest indices kept)."""
    w = workloads.make("tiny", shrink=2, steps=12)
    _run(w, policy)


@pytest.mark.parametrize("seed", [0, 1])
def test_static_top_fraction_parity(seed, cuda_device):
    w = workloads.make("llama2-13b", shrink=16, steps=14, seed=seed)
    warm, frac = 5, 0.25
    # per-unit swings during the warm-up, so the averaged GNMR separates units
    rng = np.random.default_rng(50 + seed)
    w.scales[1:warm] *= np.exp(0.3 * rng.standard_normal((warm - 1, w.num_segments)))
    state = {}

    def check(t, tr, res, got):
        if t == warm:
            # the one decision: the cut in the summed GNMR must have margin
            g = tr.ctl.policy_state()["gsum"]
            k = math.ceil(frac * w.num_units)
            top = np.sort(g)[::-1]
            assert (top[k - 1] - top[k]) > 1e-4 * top[k - 1], "no margin at the static cut"
        if t > warm:
            if "fixed" not in state:
                state["fixed"] = got["mask"].copy()
                assert got["mask"].sum() == math.ceil(frac * w.num_units)
            assert np.array_equal(got["mask"], state["fixed"])

    _run(w, dict(policy=2, static_warmup_steps=warm, static_fraction=frac), check=check)


def test_delta_mem(cuda_device):
    import oracle
    w = workloads.make("tiny", seed=4, steps=60, shrink=2)
    cost = np.random.default_rng(3).uniform(1e3, 1e6, w.num_units)

    def check(t, tr, res, got):
        want = oracle.delta_mem(res.mask, cost)
        assert got["delta_mem"][0] == pytest.approx(want, rel=1e-12, abs=0.0)
        assert got["delta_mem"][0] <= w.max_o * cost.max() * (1 + 1e-12)

    _run(w, dict(unit_cost=cost), check=check)

"""Top_maxO (Algorithm 2) on crafted risk distributions, through the
controller half (gnmr_finish), against the oracle.

Step 1 feeds n_b = 1 to every unit, so A_b = 1; from then on n_b is chosen
so that R_b = G_b / alpha takes the value a case needs (alpha = 1, beta so
large that Delta never decides, eps = 0).  The GPU and the oracle receive the
same n_b (the oracle gets sqrt of the same sums of squares) and run the same
correctly rounded fp64 operations, so R, the masks, the locks and the counts
must agree exactly -- no decision margin is needed, and ties are real.

The cases steer the selection through each of its paths.  The risk
histogram (eight bins per octave: exponent and top three mantissa bits)
locates the cut bin; its members are ranked directly (up to 512), by a radix
select in shared memory (up to 3,072), or by radix passes over the whole
candidate list in global memory (more); a cut bin can also be taken whole.
Multi-step cases drive the hot list: the previous step's prediction held
(only the hot list is read), missed (the risks fell below it), or the hot
list overflowed.  Equal risks inside the cut bin, lock-only candidates and
the admission-cap and static policies are covered too."""
import numpy as np
import pytest

import oracle
from paper_2606_00539_gb300 import Monitor

pytestmark = pytest.mark.gpu

U = 20_000
MAX_O = 64
LOCK = 2


def _spread(rng):
    return np.exp(rng.uniform(np.log(0.5), np.log(1e4), U))


def _narrow(rng):
    # [1, 1.125): one bucket of the coarse histogram (exponent and the top
    # three mantissa bits), far more members than the shared list holds
    return rng.uniform(1.0001, 1.1249, U)


def _with_cut_members(n_cut, ties=False):
    def make(rng):
        r = rng.uniform(0.5, 0.9, U)                      # not candidates
        top = rng.choice(U, 10 + n_cut, replace=False)
        r[top[:10]] = 1000.0 + np.arange(10)              # above the cut bucket
        r[top[10:]] = 8.5 if ties else rng.uniform(8.0, 9.0, n_cut)   # one bucket: [8, 9)
        return r
    return make


def _whole_bucket(rng):
    r = rng.uniform(1.3, 1.9, U)                          # candidates below the cut
    top = rng.choice(U, MAX_O, replace=False)
    r[top] = rng.uniform(96.0, 104.0, MAX_O)              # exactly maxO in one bucket: [96, 104)
    return r


CASES = {
    "spread": _spread,
    "narrow_overflow": _narrow,
    "cut_55": _with_cut_members(55),
    "cut_512": _with_cut_members(512),
    "cut_513": _with_cut_members(513),
    "cut_1500": _with_cut_members(1500),
    "cut_at_capacity": _with_cut_members(3072),
    "cut_past_capacity": _with_cut_members(3073),
    "cut_ties": _with_cut_members(300, ties=True),
    "cut_ties_radix": _with_cut_members(2000, ties=True),
    "whole_bucket": _whole_bucket,
}


def _drive(risks_per_step, policy=0, max_o=MAX_O, **policy_kw):
    """Step 1 with n = 1, then one step per entry of risks_per_step (the
    target R of every unit: n = R * A_b with A_b read from the oracle)."""
    import torch
    kw = dict(window=8, max_o=max_o, lock_len=LOCK, eps=0.0)
    mon = Monitor(np.zeros(U, np.int64), np.zeros(U, np.int64), dtype="f32", device=0,
                  alpha=1.0, beta=1e6, policy=policy, **kw, **policy_kw)
    ctl = oracle.Controller(U, alpha=(1.0, 1.0), beta=(1e6, 1e6), policy=policy, **kw, **policy_kw)
    stats = mon.new_stats()
    mask = torch.empty(U, dtype=torch.uint8, device="cuda:0")
    try:
        for t, target in enumerate([np.ones(U)] + list(risks_per_step)):
            A = ctl.get_state()["A"]
            n = np.asarray(target, np.float64) * (A if t > 0 else 1.0)
            sumsq = n * n
            mon.finish(torch.from_numpy(sumsq).to("cuda:0"), mask=mask, stats=stats)
            want = ctl.step(np.sqrt(sumsq))
            got_r = stats["risk"].cpu().numpy()
            assert np.array_equal(got_r.view(np.uint64), want.risk.view(np.uint64)), f"step {t + 1}: R"
            got_mask = mask.cpu().numpy()
            bad = np.flatnonzero(got_mask != want.mask)
            assert bad.size == 0, f"step {t + 1}: mask differs at {bad[:10]}"
            assert np.array_equal(stats["lock"].cpu().numpy(), want.lock), f"step {t + 1}: lock"
            assert stats["counts"].cpu().tolist() == [want.n_candidates, want.n_selected], \
                f"step {t + 1}: counts"
    finally:
        mon.close()
        ctl.close()
    return want


@pytest.mark.parametrize("case", sorted(CASES))
def test_top_max_o_paths(case, cuda_device):
    rng = np.random.default_rng(sorted(CASES).index(case) + 101)
    res = _drive([CASES[case](rng)])
    assert res.n_selected == MAX_O


def _scaled(factor):
    def make(rng):
        return _spread(rng) * factor
    return make


HOT_SEQUENCES = {
    # the same distribution every step: from step 3 on the prediction holds
    "stationary": [_spread] * 5,
    # risks shift down by 100x: the cut falls below the predicted bin (full list)
    "shift_down": [_spread, _spread, _scaled(0.01), _scaled(0.01), _spread],
    # risks shift up by 100x: the cut rises above the prediction (hot list holds more)
    "shift_up": [_spread, _spread, _scaled(100.0), _spread],
    # a step whose pool fits the budget (every candidate hot next step), then a
    # step with ~20,000 candidates: the hot list overflows (full list)
    "overflow": [lambda rng: np.full(U, 0.5), _with_cut_members(20, ties=False), _narrow, _spread],
    # a cut bin ranked by the shared-memory radix select out of the hot list
    "hot_radix": [_with_cut_members(1500), _with_cut_members(1500), _with_cut_members(1500)],
}


@pytest.mark.parametrize("seq", sorted(HOT_SEQUENCES))
def test_hot_list_predictions(seq, cuda_device):
    rng = np.random.default_rng(sorted(HOT_SEQUENCES).index(seq) + 301)
    _drive([make(rng) for make in HOT_SEQUENCES[seq]])


def test_lock_only_candidates_compete_with_new_spikes(cuda_device):
    """Step 2 selects maxO units (Lock = T_lock); at step 3 they fall to
    R <= 1 but stay candidates through their locks, competing with 30 new
    spikes: the spikes win, and the highest lock-only risks fill the rest."""
    rng = np.random.default_rng(7)
    r2 = _spread(rng)
    r3 = rng.uniform(0.2, 0.95, U)
    spikes = rng.choice(U, 30, replace=False)
    r3[spikes] = rng.uniform(5.0, 50.0, 30)
    res = _drive([r2, r3, rng.uniform(0.2, 0.95, U)])
    assert res.n_candidates > 0


def test_admission_cap_counts_only_new_units(cuda_device):
    """Under the admission cap the histogram holds only the units not active
    at t - 1; retained units pass outside the cap."""
    rng = np.random.default_rng(8)
    steps = [_spread(rng) for _ in range(4)]
    _drive(steps, policy=oracle.POLICY_ADMISSION_CAP)


def test_admission_cap_retained_past_the_hot_list_capacity(cuda_device):
    """Admission cap with a budget of 5,000: the admitted units stay active
    (their locks keep them candidates), so by the fourth step more than
    8,192 retained units have to join the hot list, which overflows; the
    selection then reads the whole candidate list."""
    rng = np.random.default_rng(10)
    res = _drive([_spread(rng) for _ in range(5)], policy=oracle.POLICY_ADMISSION_CAP, max_o=5000)
    assert res.n_selected > 8192


def test_static_policy_ranks_by_gnmr_sum(cuda_device):
    """The static policy ranks every recoverable unit once, by its GNMR sum
    over the warm-up (here steps 1-2), keeping ceil(0.01 |B_rec|) units."""
    rng = np.random.default_rng(9)
    steps = [_spread(rng), rng.uniform(0.5, 2.0, U), rng.uniform(0.5, 2.0, U)]
    _drive(steps, policy=oracle.POLICY_STATIC_TOP, static_warmup_steps=2, static_fraction=0.01)


def _random_sums(rng, U, t, prev):
    """Per-unit sums of squares for one step: spread values with exact zeros,
    exact repeats of the previous step (equal risks), a few spikes and, now
    and then, an infinite sum (a non-finite gradient)."""
    s = np.exp(rng.normal(0.0, 1.0, U))
    kind = rng.random(U)
    s[kind < 0.10] = 0.0
    if prev is not None:
        rep = kind > 0.85
        s[rep] = prev[rep]
    spikes = rng.random(U) < 0.05
    s[spikes] *= rng.uniform(10.0, 1e4, int(spikes.sum()))
    if t > 2 and rng.random() < 0.2:
        s[rng.integers(0, U)] = np.inf
    return s


@pytest.mark.parametrize("seed", range(64))
def test_random_small_controllers_agree_exactly(seed, cuda_device):
    """Random small configurations through the controller half: the unit
    count, window, maxO (0, below and above U), T_lock, policy, thresholds
    (some below 1, so risks tie at t = 1) and eps vary; sums include zeros,
    repeats and infinities.  The GPU and the oracle get the same n_b and run
    the same IEEE fp64 operations, so R, masks, locks and counts agree bit
    for bit at every step."""
    import torch
    rng = np.random.default_rng(1000 + seed)
    U = int(rng.integers(1, 200))
    policy = int(rng.integers(0, 3))
    kw = dict(window=int(rng.integers(1, 10)), max_o=int(rng.choice([0, 1, 3, max(1, U // 4), U, U + 2])),
              lock_len=int(rng.integers(0, 5)), eps=float(rng.choice([0.0, 1e-8])))
    a = tuple(float(x) for x in rng.choice([0.9, 1.1, 1.5, 2.0], 2))
    b = tuple(float(x) for x in rng.choice([0.8, 1.3, 1.5], 2))
    warm = int(rng.integers(0, 4))
    pol = dict(policy=policy, forced_recovery_steps=int(rng.integers(0, 3)) if policy != 2 else 0,
               static_warmup_steps=int(rng.integers(0, 4)) if policy == 2 else 0,
               static_fraction=float(rng.choice([0.1, 0.25, 0.5])))
    rec = (rng.random(U) < 0.8).astype(np.uint8)
    mon = Monitor(np.zeros(U, np.int64), np.zeros(U, np.int64), dtype="f32", device=0, alpha=a, beta=b,
                  warmup_steps=warm, recoverable=rec, **kw, **pol)
    ctl = oracle.Controller(U, alpha=a, beta=b, warmup_steps=warm, recoverable=rec, **kw, **pol)
    stats = mon.new_stats()
    mask = torch.empty(U, dtype=torch.uint8, device="cuda:0")
    prev = None
    try:
        for t in range(12):
            sumsq = _random_sums(rng, U, t, prev)
            prev = sumsq
            mon.finish(torch.from_numpy(sumsq).to("cuda:0"), mask=mask, stats=stats)
            want = ctl.step(np.sqrt(sumsq))
            got_r = stats["risk"].cpu().numpy()
            assert np.array_equal(got_r.view(np.uint64), want.risk.view(np.uint64)), f"step {t + 1}: R"
            assert np.array_equal(mask.cpu().numpy(), want.mask), f"step {t + 1}: mask"
            assert np.array_equal(stats["lock"].cpu().numpy(), want.lock), f"step {t + 1}: lock"
            assert stats["counts"].cpu().tolist() == [want.n_candidates, want.n_selected], f"step {t + 1}: counts"
    finally:
        mon.close()
        ctl.close()

"""Pins for the CPU oracle: each test checks the oracle against something other
than itself -- hand-derived traces, closed forms, library routines, brute
force and the invariants the paper states -- chosen so that a dropped term, a
wrong sign or index, or a swapped operand in the oracle fails at least one.
"""
import itertools
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests.golden import hand_traces

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _f(x):
    return float(x)


def policy_kwargs(cfg):
    return dict(policy=int(cfg.get("policy", 0)), forced_recovery_steps=int(cfg.get("forced", 0)),
                static_warmup_steps=int(cfg.get("static_warmup", 0)),
                static_fraction=_f(cfg.get("static_fraction", Fraction(1, 4))))


def _controller_from(cfg):
    return oracle.Controller(
        int(cfg["units"]), int(cfg["window"]), int(cfg["max_o"]), int(cfg["lock_len"]),
        alpha=(_f(cfg["alpha_init"]), _f(cfg["alpha_main"])),
        beta=(_f(cfg["beta_init"]), _f(cfg["beta_main"])),
        warmup_steps=int(cfg["warmup"]), eps=_f(cfg["eps"]),
        recoverable=np.array([int(x) for x in cfg["recoverable"]], np.uint8),
        **policy_kwargs(cfg))


def _close(got, want, rel=1e-12):
    want = float(want)
    if math.isinf(want):
        return got == want
    return abs(got - want) <= rel * max(1.0, abs(want))


# ---------------------------------------------------------------------------
# Hand-derived traces (Algorithm 1 and Algorithm 2, exact rationals)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("trace", hand_traces.all_traces(), ids=lambda t: t.name)
def test_hand_trace(trace):
    ctl = _controller_from(trace.cfg)
    U = int(trace.cfg["units"])
    for st in trace.steps:
        res = ctl.step(np.array([float(x) for x in st.n]))
        state = ctl.get_state()
        for b in range(U):
            assert _close(res.gnmr[b], st.gnmr[b]), (st.t, b, "GNMR")
            assert _close(res.dgnmr[b], st.dgnmr[b]), (st.t, b, "Delta-GNMR")
            assert _close(res.risk[b], st.risk[b]), (st.t, b, "R")
            assert _close(state["A"][b], st.mean_after[b]), (st.t, b, "A")
        assert res.n_candidates == len(st.candidates), st.t
        assert res.n_selected == len(st.selected), st.t
        assert list(np.nonzero(res.mask)[0]) == st.selected, st.t
        assert list(res.lock) == st.lock_after, st.t
        assert state["t"] == st.t


def test_hand_trace_fixtures_are_consistent():
    """The fixtures themselves: R = max(G/alpha, D/beta) and the candidate
    sets follow from R and the previous locks, with exact rationals."""
    for tr in hand_traces.all_traces():
        cfg = tr.cfg
        prev_lock = [0] * int(cfg["units"])
        for st in tr.steps:
            a = cfg["alpha_init"] if st.t <= cfg["warmup"] else cfg["alpha_main"]
            b_ = cfg["beta_init"] if st.t <= cfg["warmup"] else cfg["beta_main"]
            for b in range(int(cfg["units"])):
                g, d = st.gnmr[b], st.dgnmr[b]
                r = max(g / a if not isinstance(g, float) else g,
                        d / b_ if not isinstance(d, float) else d)
                assert r == st.risk[b], (tr.name, st.t, b)
            pool_formed = st.t > cfg.get("forced", 0) and cfg.get("policy", 0) != 2
            if pool_formed:
                cand = [b for b in range(int(cfg["units"]))
                        if cfg["recoverable"][b] and (st.risk[b] > 1 or prev_lock[b] > 0)]
                assert cand == st.candidates, (tr.name, st.t)
            prev_lock = st.lock_after


# ---------------------------------------------------------------------------
# Norms (Eq. local_gradient) against library routines and closed forms
# ---------------------------------------------------------------------------

def test_norm_bf16_decode_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 1 << 16, size=4096, dtype=np.uint32).astype(np.uint16)
    exp = (bits >> 7) & 0xFF
    bits = bits[exp != 0xFF]                      # drop NaN/Inf patterns
    off = np.arange(len(bits), dtype=np.int64)
    ln = np.ones(len(bits), dtype=np.int64)
    got = oracle.unit_norms(bits, off, ln)
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).float().double().abs()
    assert np.array_equal(got, ref.numpy())


def test_norm_matches_fsum_fp32():
    rng = np.random.default_rng(2)
    x = (rng.standard_normal(50_000) * np.exp(rng.standard_normal(50_000))).astype(np.float32)
    off = np.array([0, 17, 1000, 49_999, 3], np.int64)
    ln = np.array([50_000, 983, 12_345, 1, 0], np.int64)
    got = oracle.unit_norms(x, off, ln)
    for b in range(len(off)):
        seg = x[off[b]:off[b] + ln[b]].astype(np.float64)
        exact = math.sqrt(math.fsum(seg * seg))           # correctly rounded sum
        assert got[b] == pytest.approx(exact, rel=1e-12, abs=0.0)
        assert got[b] == pytest.approx(np.linalg.norm(seg), rel=1e-12, abs=0.0)


def test_norm_special_values():
    ones = np.ones(1 << 20, np.float32)
    zeros = np.zeros(1000, np.float32)
    got = oracle.unit_norms(ones, [0, 5, 0], [1 << 20, 1 << 16, 0])
    assert got[0] == 1024.0 and got[1] == 256.0 and got[2] == 0.0
    assert oracle.unit_norms(zeros, [0], [1000])[0] == 0.0
    # Signs do not matter; a power-of-two scale is exact.
    rng = np.random.default_rng(3)
    x = rng.standard_normal(777).astype(np.float32)
    base = oracle.unit_norms(x, [0], [777])[0]
    assert oracle.unit_norms(-x, [0], [777])[0] == base
    assert oracle.unit_norms(x * np.float32(8.0), [0], [777])[0] == 8.0 * base


def test_segmented_norm_is_the_norm_of_the_concatenation():
    """A block unit's norm (Sec. 3.4) is the L2 norm of all its segments'
    elements together: compared with fsum over the concatenation."""
    rng = np.random.default_rng(4)
    x = (rng.standard_normal(20_000) * np.exp(2 * rng.standard_normal(20_000))).astype(np.float32)
    off = np.array([0, 5000, 100, 7000, 19_000, 3, 12_000], np.int64)
    ln = np.array([100, 2000, 900, 0, 1000, 4, 5000], np.int64)
    unit = np.array([2, 0, 2, 1, 0, 2, 4], np.int32)          # unit 3 has no segment
    for threads in (1, 3):
        got = oracle.unit_norms_segmented(x, off, ln, unit, 5, threads)
        for b in range(5):
            seg = np.concatenate([x[o:o + n] for o, n, u in zip(off, ln, unit) if u == b] +
                                 [np.zeros(0, np.float32)]).astype(np.float64)
            assert got[b] == pytest.approx(math.sqrt(math.fsum(seg * seg)), rel=1e-12, abs=0.0)
        assert got[3] == 0.0 and got[1] == 0.0
    # one segment per unit: the plain per-unit norm
    ident = np.arange(len(off), dtype=np.int32)
    assert np.allclose(oracle.unit_norms_segmented(x, off, ln, ident, len(off)),
                       oracle.unit_norms(x, off, ln), rtol=1e-15, atol=0)


def test_delta_mem_is_the_cost_of_the_active_set():
    """Eq. generic-memory-bound: Delta M_t = sum of c_b over b in A_t, at most
    maxO * c_max under the active cap."""
    rng = np.random.default_rng(12)
    U = 40
    cost = rng.uniform(1, 100, U)
    ctl = oracle.Controller(U, 3, 5, 2, alpha=(1.05, 1.05), beta=(1.05, 1.05))
    for norms in _spiky_trace(rng, 30, U, spike_p=0.3):
        res = ctl.step(norms)
        dm = oracle.delta_mem(res.mask, cost)
        assert dm == pytest.approx(math.fsum(cost[b] for b in range(U) if res.mask[b]), rel=1e-15)
        assert dm <= 5 * cost.max()


def test_norm_nonfinite_propagates():
    x = np.ones(10, np.float32)
    x[3] = np.inf
    y = np.ones(10, np.float32)
    y[4] = np.nan
    assert math.isinf(oracle.unit_norms(x, [0], [10])[0])
    assert math.isnan(oracle.unit_norms(y, [0], [10])[0])


# ---------------------------------------------------------------------------
# Algorithm 1 against the closed forms of Sec. 3.1-3.2 (batch, eps = 0)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("window", [1, 3, 8])
def test_algorithm1_matches_closed_forms(window):
    rng = np.random.default_rng(10 + window)
    T, U = 40, 5
    n = np.exp(rng.standard_normal((T, U)))
    ctl = oracle.Controller(U, window, 2, 3, alpha=(1.3, 1.3), beta=(1.2, 1.2), eps=0.0)
    G_hist = np.zeros((T, U))
    for t in range(T):
        res = ctl.step(n[t])
        # GNMR_t = n_t / ((1/(t-1)) sum_{tau<t} n_tau), GNMR_1 = 1 (Eq. GNMR).
        want_g = np.ones(U) if t == 0 else n[t] / n[:t].mean(axis=0)
        np.testing.assert_allclose(res.gnmr, want_g, rtol=1e-12)
        # Delta-GNMR_t = GNMR_t / ((1/delta) sum_{tau=1..delta} GNMR_{t-tau}),
        # and 1 until delta past values exist (Eq. Delta-GNMR, Alg. 1).
        want_d = np.ones(U) if t < window else want_g / G_hist[t - window:t].mean(axis=0)
        np.testing.assert_allclose(res.dgnmr, want_d, rtol=1e-12)
        G_hist[t] = want_g
        # A_t is the plain arithmetic mean of n_1..n_t.
        np.testing.assert_allclose(ctl.get_state()["A"], n[:t + 1].mean(axis=0), rtol=1e-12)
        np.testing.assert_allclose(res.risk, np.maximum(want_g / 1.3, want_d / 1.2), rtol=1e-12)


def test_eps_enters_both_denominators():
    eps = 0.25
    ctl = oracle.Controller(1, 1, 1, 0, eps=eps)
    ctl.step(np.array([2.0]))
    r = ctl.step(np.array([3.0]))
    assert r.gnmr[0] == pytest.approx(3.0 / (2.0 + eps), rel=1e-15)
    assert r.dgnmr[0] == pytest.approx((3.0 / (2.0 + eps)) / (1.0 + eps), rel=1e-15)


# ---------------------------------------------------------------------------
# Algorithm 2: brute force over subsets and the invariants of Sec. 3.3
# ---------------------------------------------------------------------------

def _brute_force_selection(risk, cand, max_o):
    """Cor. 1: with a modular objective any top-k maximises the summed score;
    among maximisers take the lexicographically smallest index tuple."""
    k = min(max_o, len(cand))
    best = None
    for sub in itertools.combinations(sorted(cand), k):
        key = (sum(Fraction(risk[b]) for b in sub), tuple(-b for b in sub))
        if best is None or key > best[0]:
            best = (key, sub)
    return set(best[1]) if best else set()


@pytest.mark.parametrize("seed", range(40))
def test_algorithm2_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    U = int(rng.integers(1, 7))
    max_o = int(rng.integers(0, U + 2))
    lock_len = int(rng.integers(0, 4))
    thr = float(rng.choice([0.75, 1.0, 1.25, 1.5]))
    rec = (rng.random(U) < 0.8).astype(np.uint8)
    ctl = oracle.Controller(U, 2, max_o, lock_len, alpha=(thr, thr), beta=(thr, thr),
                            eps=0.0, recoverable=rec)
    lock_prev = np.zeros(U, np.int32)
    for _ in range(12):
        norms = rng.choice([0.5, 1.0, 2.0, 3.0], size=U)     # coarse values make ties
        res = ctl.step(norms)
        cand = [b for b in range(U) if rec[b] and (res.risk[b] > 1 or lock_prev[b] > 0)]
        assert res.n_candidates == len(cand)
        sel = _brute_force_selection(res.risk, cand, max_o)
        assert set(np.nonzero(res.mask)[0]) == sel
        for b in range(U):
            if not rec[b] or b not in sel:
                want = 0
            elif res.risk[b] > 1:
                want = lock_len
            else:
                want = max(lock_prev[b] - 1, 0)
            assert res.lock[b] == want
        lock_prev = res.lock.copy()


def _spiky_trace(rng, T, U, spike_p=0.05):
    s = np.exp(rng.standard_normal(U))
    out = []
    for _ in range(T):
        s = s * np.exp(0.05 * rng.standard_normal(U))
        f = np.where(rng.random(U) < spike_p, np.exp(rng.uniform(np.log(2), np.log(50), U)), 1.0)
        out.append(s * f * (1 + 0.02 * rng.standard_normal(U)))
    return np.array(out)


@pytest.mark.parametrize("seed", range(6))
def test_algorithm2_invariants(seed):
    rng = np.random.default_rng(200 + seed)
    U, T = 60, 80
    max_o, lock_len, window = 4, 3, 5
    rec = (rng.random(U) < 0.85).astype(np.uint8)
    ctl = oracle.Controller(U, window, max_o, lock_len, alpha=(1.5, 1.1), beta=(1.3, 1.3),
                            warmup_steps=5, eps=1e-8, recoverable=rec)
    lock_prev = np.zeros(U, np.int32)
    for t, norms in enumerate(_spiky_trace(rng, T, U)):
        res = ctl.step(norms)
        sel = np.nonzero(res.mask)[0]
        cand = [b for b in range(U) if rec[b] and (res.risk[b] > 1 or lock_prev[b] > 0)]
        assert len(sel) <= max_o                                    # |A_t| <= maxO
        assert set(sel) <= set(cand)                                # A_t within C_t
        assert all(rec[b] for b in cand)                            # C_t within B_rec
        assert len(sel) == min(max_o, len(cand))                    # cap, not a target
        assert np.all((res.lock >= 0) & (res.lock <= lock_len))
        assert np.all(res.mask[res.lock > 0] == 1)                  # Lock > 0 only if selected
        assert np.all(res.lock[rec == 0] == 0) and np.all(res.mask[rec == 0] == 0)
        if t == 0:
            assert np.all(res.gnmr == 1.0)                          # GNMR_1 = 1
        if t < window:
            assert np.all(res.dgnmr == 1.0)                         # |Q| < delta
        unsel = [b for b in cand if not res.mask[b]]
        if len(sel) and unsel:
            assert min(res.risk[sel]) >= max(res.risk[unsel])       # Top_maxO order
        hot = [b for b in cand if res.risk[b] > 1]
        lock_only = [b for b in cand if res.risk[b] <= 1]
        if lock_only and any(res.mask[b] for b in lock_only):
            assert all(res.mask[b] for b in hot)                    # R > 1 outranks locks
        lock_prev = res.lock.copy()


def test_plain_threshold_special_case():
    """maxO >= U and T_lock = 0: the mask is exactly {b recoverable : R > 1}."""
    rng = np.random.default_rng(5)
    U = 30
    rec = (rng.random(U) < 0.7).astype(np.uint8)
    ctl = oracle.Controller(U, 4, U, 0, alpha=(1.2, 1.2), beta=(1.2, 1.2), recoverable=rec)
    for norms in _spiky_trace(rng, 50, U, spike_p=0.2):
        res = ctl.step(norms)
        assert np.array_equal(res.mask, ((res.risk > 1) & (rec == 1)).astype(np.uint8))


def test_constant_norms_never_trigger():
    ctl = oracle.Controller(8, 3, 8, 5, alpha=(1.01, 1.01), beta=(1.01, 1.01), eps=0.0)
    norms = np.array([0.5, 1, 2, 3, 1e-3, 1e3, 7, 9], float)
    for _ in range(30):
        res = ctl.step(norms)
        assert np.all(res.gnmr == 1.0) and np.all(res.dgnmr == 1.0)
        assert res.n_candidates == 0 and not res.mask.any()


def test_per_unit_scale_invariance():
    """GNMR and Delta-GNMR are dimensionless: scaling one unit's norms by a
    constant at every step leaves them unchanged (eps = 0)."""
    rng = np.random.default_rng(6)
    U, T = 10, 40
    tr = _spiky_trace(rng, T, U, spike_p=0.1)
    scale = np.array([1, 2.0 ** 10, 3.7, 1e-4, 1, 1, 5e5, 1, 0.3, 1])
    a = oracle.Controller(U, 4, 3, 2, eps=0.0)
    b = oracle.Controller(U, 4, 3, 2, eps=0.0)
    for norms in tr:
        ra, rb = a.step(norms), b.step(norms * scale)
        np.testing.assert_allclose(ra.gnmr, rb.gnmr, rtol=1e-12)
        np.testing.assert_allclose(ra.dgnmr, rb.dgnmr, rtol=1e-12)
        assert np.array_equal(ra.mask, rb.mask)


def test_nonfinite_norm_reading():
    ctl = oracle.Controller(3, 2, 1, 2, eps=0.0)
    for _ in range(3):
        ctl.step(np.array([1.0, 1.0, 1.0]))
    before = ctl.get_state()
    res = ctl.step(np.array([np.nan, 1.0, np.inf]))
    after = ctl.get_state()
    assert math.isinf(res.risk[0]) and math.isinf(res.risk[2])
    assert list(np.nonzero(res.mask)[0]) == [0]          # tie at +inf, lower index
    for key in ("A", "k", "Q", "qlen"):
        assert np.array_equal(before[key][[0, 2]], after[key][[0, 2]])
    assert after["k"][1] == before["k"][1] + 1


def test_checkpoint_resume_is_seamless():
    rng = np.random.default_rng(7)
    U, T = 12, 30
    tr = _spiky_trace(rng, T, U, spike_p=0.15)
    full = oracle.Controller(U, 3, 2, 2)
    part = oracle.Controller(U, 3, 2, 2)
    masks_full = [full.step(n).mask for n in tr]
    for n in tr[:13]:
        part.step(n)
    resumed = oracle.Controller(U, 3, 2, 2)
    resumed.set_state(part.get_state())
    masks_res = [resumed.step(n).mask for n in tr[13:]]
    for a, b in zip(masks_full[13:], masks_res):
        assert np.array_equal(a, b)


def test_gnmr_exceedance_decreases_on_iid_norms():
    """Theorem 2 (Sec. 4): for iid sub-exponential norms the probability that
    GNMR_t >= alpha falls as the history grows.  A statistical smoke check."""
    rng = np.random.default_rng(8)
    U, T = 2000, 60
    ctl = oracle.Controller(U, 4, 0, 0, eps=0.0)
    hits = np.zeros(T)
    for t in range(T):
        res = ctl.step(rng.exponential(1.0, U) + 1.0)
        hits[t] = np.mean(res.gnmr >= 1.6)
    assert hits[1:5].mean() > hits[40:].mean()


@pytest.mark.parametrize("seed", range(6))
def test_admission_cap_invariants(seed):
    """Remark on the maxO budget: only newly admitted units are capped."""
    rng = np.random.default_rng(300 + seed)
    U, max_o = 30, 3
    rec = (rng.random(U) < 0.8).astype(np.uint8)
    ctl = oracle.Controller(U, 3, max_o, 2, alpha=(1.1, 1.1), beta=(1.1, 1.1), recoverable=rec,
                            policy=oracle.POLICY_ADMISSION_CAP)
    prev_active = np.zeros(U, bool)
    lock_prev = np.zeros(U, np.int32)
    for norms in _spiky_trace(rng, 40, U, spike_p=0.2):
        res = ctl.step(norms)
        A = res.mask.astype(bool)
        cand = np.array([bool(rec[b]) and (res.risk[b] > 1 or lock_prev[b] > 0) for b in range(U)])
        assert not np.any(A & ~cand)                               # A_t within C_t
        assert np.all(A[cand & prev_active])                       # retained
        new = cand & ~prev_active
        admitted = np.nonzero(A & new)[0]
        assert len(admitted) == min(max_o, int(new.sum()))         # |S_t| <= maxO, filled
        rest = [b for b in np.nonzero(new)[0] if b not in admitted]
        if len(admitted) and rest:                                 # the best new ones by R
            worst = min(admitted, key=lambda b: (res.risk[b], -b))
            best_rest = max(rest, key=lambda b: (res.risk[b], -b))
            assert (res.risk[worst], -worst) > (res.risk[best_rest], -best_rest)
        assert res.n_selected == int(A.sum())
        prev_active = A
        lock_prev = res.lock.copy()


@pytest.mark.parametrize("n_forced,n_static", [(5, 6), (1, 1), (0, 0)])
def test_forced_and_static_policies(n_forced, n_static):
    """Forced warm-up: every recoverable unit selected for t <= n_forced.
    Static policy: every recoverable unit selected for t <= n_static, then
    the ceil(0.3 |B_rec|) largest GNMR sums over those steps (ties by index;
    with no warm-up all sums are 0) for good.  A one-step warm-up is the
    case where the all-on steps cannot lean on state left by an earlier
    all-on step."""
    rng = np.random.default_rng(17)
    U, T = 20, 25
    rec = (rng.random(U) < 0.7).astype(np.uint8)
    tr = _spiky_trace(rng, T, U, spike_p=0.2)
    base = oracle.Controller(U, 3, 4, 2, recoverable=rec)
    forced = oracle.Controller(U, 3, 4, 2, recoverable=rec, forced_recovery_steps=n_forced)
    stat = oracle.Controller(U, 3, 4, 2, recoverable=rec, policy=oracle.POLICY_STATIC_TOP,
                             static_warmup_steps=n_static, static_fraction=0.3)
    gsum = np.zeros(U)
    fixed = None
    for t, norms in enumerate(tr, start=1):
        rb, rf, rs = base.step(norms), forced.step(norms), stat.step(norms)
        # the policies never change the statistics
        np.testing.assert_array_equal(rb.gnmr, rf.gnmr)
        np.testing.assert_array_equal(rb.gnmr, rs.gnmr)
        if t <= n_forced:
            assert np.array_equal(rf.mask, rec) and rf.n_selected == rec.sum()
        else:
            np.testing.assert_array_equal(rf.risk, rb.risk)
        if t <= n_static:
            assert np.array_equal(rs.mask, rec)
            gsum += np.where(rec == 1, rb.gnmr, 0.0)
        else:
            if fixed is None:
                k = math.ceil(0.3 * rec.sum())
                order = sorted(np.nonzero(rec)[0], key=lambda b: (-gsum[b], b))
                fixed = np.zeros(U, np.uint8)
                fixed[order[:k]] = 1
            assert np.array_equal(rs.mask, fixed)
            assert np.all(rs.lock == 0)

"""Runs a workload through the CUDA path and the oracle in lockstep.

Each step: the fill kernel writes the step's gradients, the oracle computes
the norms from the same bytes (copied to the host) and Algorithms 1 and 2.
Before the GPU step runs, every decision that depends on a rounded quantity is
checked for margin (R at least 1e-3 away from 1; the maxO-th and (maxO+1)-th
risk at least 1e-3 apart); a unit that lacks margin gets its scale multiplied
by a keyed redraw within +-1 % and is regenerated.  Values that the method
computes exactly on both sides (GNMR = 1 on a first step or zero mean,
Delta-GNMR = 1 while the window fills, zero norms, +inf) need no margin.
"""
from __future__ import annotations

import math
import os
from dataclasses import dataclass, field

import numpy as np

import oracle
import workloads

MARGIN = 1e-3
MAX_ATTEMPTS = 12


def _thresholds(w, t, alpha=math.nan, beta=math.nan):
    a_t = alpha if not math.isnan(alpha) else (w.alpha[0] if t <= w.warmup_steps else w.alpha[1])
    b_t = beta if not math.isnan(beta) else (w.beta[0] if t <= w.warmup_steps else w.beta[1])
    return a_t, b_t


def _exactness(state, res, w, t, alpha=math.nan, beta=math.nan):
    """Per unit: is R computed exactly (identically by both implementations)?"""
    a_t, b_t = _thresholds(w, t, alpha, beta)
    g_exact = (state["k"] == 0) | (state["A"] == 0.0) | (res.gnmr == 0.0) | np.isinf(res.gnmr)
    d_exact = (state["qlen"] < w.window) | (res.dgnmr == 0.0) | np.isinf(res.dgnmr)
    x, y = res.gnmr / a_t, res.dgnmr / b_t
    exact = (g_exact & d_exact) | (g_exact & (x > y * (1 + MARGIN))) | (d_exact & (y > x * (1 + MARGIN)))
    return exact


def margin_violations(state_before, res, w, t, alpha=math.nan, beta=math.nan, policy=None,
                      active_before=None):
    """Units whose GPU decision could differ from the oracle's by rounding.
    ``w`` needs alpha, beta, warmup_steps, window, max_o and recoverable;
    ``policy`` (dict of the policy settings) and ``active_before`` (A_{t-1})
    for the policy variants."""
    policy = policy or {}
    forced = policy.get("forced_recovery_steps", 0)
    kind = policy.get("policy", 0)
    warm = policy.get("static_warmup_steps", 0)
    if t <= forced or (kind == 2 and t <= warm):
        return []                                   # no decision depends on a rounded value
    rec = np.asarray(w.recoverable).astype(bool)
    if kind == 2:
        return []                                   # the static choice is checked separately
    exact = _exactness(state_before, res, w, t, alpha, beta)
    r = res.risk
    bad = set(np.nonzero(rec & ~exact & (np.abs(r - 1.0) < MARGIN))[0].tolist())
    lock_prev = state_before["lock"]
    cand = np.nonzero(rec & ((r > 1.0) | (lock_prev > 0)))[0]
    if kind == 1 and active_before is not None:    # the cap applies to new candidates only
        cand = np.array([b for b in cand if not active_before[b]], dtype=np.int64)
    if len(cand) > w.max_o and w.max_o > 0:
        order = sorted(cand.tolist(), key=lambda b: (-r[b], b))
        a, b = order[w.max_o - 1], order[w.max_o]
        if not (exact[a] and exact[b]):
            if r[a] - r[b] < MARGIN * r[a]:
                bad.update(x for x in (a, b) if not exact[x])
    # Noisy units exactly at the same value as an exact one cannot occur
    # (margin above); ties between noisy units are covered by the cut check.
    return sorted(bad)


@dataclass
class StepRecord:
    t: int
    attempts: int
    repaired: list = field(default_factory=list)


class LockstepTrace:
    """Drives one workload on the GPU monitor and the oracle."""

    def __init__(self, w: workloads.Workload, device, monitor_factory, threads: int = 0,
                 policy: dict | None = None):
        import torch
        self.torch = torch
        self.w = w
        self.dev = torch.device(device)
        self.filler = workloads.Filler(w, self.dev)
        self.arena = self.filler.new_arena()
        self.policy = dict(policy or {})
        self.mon = monitor_factory(w, **self.policy) if self.policy else monitor_factory(w)
        ctl_policy = {k: v for k, v in self.policy.items() if k != "unit_cost"}
        self.ctl = oracle.Controller(w.num_units, **w.controller_kwargs(), **ctl_policy)
        self.stats = self.mon.new_stats()
        self.threads = threads or min(16, os.cpu_count() or 1)
        self.records = []
        self._pinned = None
        if self.arena.numel() * self.arena.element_size() > (256 << 20):
            # large arenas: one reusable pinned host copy instead of a fresh
            # pageable allocation every step
            self._pinned = torch.empty(self.arena.numel(), dtype=self.arena.dtype, pin_memory=True)

    def close(self):
        self.mon.close()
        self.ctl.close()

    def _host_norms(self, units=None):
        torch = self.torch
        w = self.w
        torch.cuda.synchronize(self.dev)
        if units is None or w.segment_unit is not None:
            if self._pinned is not None:
                self._pinned.copy_(self.arena)
                host = self._pinned
            else:
                host = self.arena.cpu()
            view = host.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16" else host.numpy()
            if w.segment_unit is not None:
                n = oracle.unit_norms_segmented(view, w.offsets, w.lengths, w.segment_unit,
                                                w.num_units, self.threads)
                return n if units is None else {u: n[u] for u in units}
            return oracle.unit_norms_threaded(view, w.offsets, w.lengths, self.threads)
        out = {}
        for u in units:
            o, n = int(w.offsets[u]), int(w.lengths[u])
            seg = self.arena[o:o + n].cpu()
            view = seg.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16" else seg.numpy()
            out[u] = oracle.unit_norms(view, [0], [n])[0]
        return out

    def step(self, t, alpha=math.nan, beta=math.nan, gpu_step=None):
        """Generates step t with margin repair, advances the oracle (with the
        given threshold overrides), runs the GPU step (``gpu_step()`` if given,
        which must write self.stats and return the mask) and returns
        (oracle norms, oracle result, GPU outputs as numpy)."""
        w = self.w
        scales = w.scales[t].copy()                       # per segment (tensor)
        attempts = np.zeros(w.num_segments, np.int32)
        unit_attempts = np.zeros(w.num_units, np.int32)
        self.filler.fill(self.arena, t, scales, attempts)
        norms = self._host_norms()
        rec = StepRecord(t + 1, 0)
        while True:
            before = self.ctl.get_state()
            policy_before = self.ctl.policy_state()
            active_before = policy_before["active"]
            res = self.ctl.step(norms, alpha, beta)
            bad = margin_violations(before, res, w, t + 1, alpha, beta, self.policy, active_before)
            if not bad:
                break
            if rec.attempts >= MAX_ATTEMPTS:
                raise RuntimeError(f"step {t + 1}: no margin after {MAX_ATTEMPTS} redraws: {bad[:8]}")
            self.ctl.set_state(before)
            self.ctl.set_policy_state(policy_before)
            rec.attempts += 1
            segs = []
            for u in bad:                                  # one factor for all of a unit's tensors
                unit_attempts[u] += 1
                f = workloads.redraw_factor(w.seed, u, t, int(unit_attempts[u]))
                mine = [u] if w.segment_unit is None else np.nonzero(w.segment_unit == u)[0].tolist()
                for g in mine:
                    attempts[g] += 1
                    scales[g] *= f
                segs.extend(mine)
            rec.repaired.extend(bad)
            self.filler.fill(self.arena, t, scales, attempts, units=segs)
            for u, v in self._host_norms(bad).items():
                norms[u] = v
        self.records.append(rec)
        if gpu_step is None:
            mask = self.mon.step(self.arena, stats=self.stats)
        else:
            mask = gpu_step()
        self.torch.cuda.synchronize(self.dev)
        got = {k: v.cpu().numpy() for k, v in self.stats.items()}
        got["mask"] = mask.cpu().numpy()
        return norms, res, got


def compare(norms, res, got, rtol=1e-5):
    """Asserts GPU == oracle: masks, locks and counts exactly, norms and
    ratios to a relative rtol (inf and NaN must match in place)."""
    def close(a, b, what):
        a = np.asarray(a, np.float64)
        b = np.asarray(b, np.float64)
        for kind, f in (("inf", np.isposinf), ("-inf", np.isneginf), ("nan", np.isnan)):
            same = f(a) == f(b)
            assert same.all(), f"{what}: {kind} pattern differs at {np.nonzero(~same)[0][:8]}"
        fin = np.isfinite(b)
        err = np.abs(a[fin] - b[fin])
        ok = err <= rtol * np.abs(b[fin])
        assert ok.all(), (f"{what}: max rel err "
                          f"{np.max(err / np.maximum(np.abs(b[fin]), 1e-300)):.3e} at "
                          f"{np.nonzero(fin)[0][~ok][:8]}")
    close(got["norm"], norms, "norm")
    close(got["gnmr"], res.gnmr, "GNMR")
    close(got["dgnmr"], res.dgnmr, "Delta-GNMR")
    close(got["risk"], res.risk, "R")
    diff = np.nonzero(got["mask"] != res.mask)[0]
    assert diff.size == 0, f"mask differs at units {diff[:16]}"
    diff = np.nonzero(got["lock"] != res.lock)[0]
    assert diff.size == 0, f"lock differs at units {diff[:16]}"
    assert list(got["counts"]) == [res.n_candidates, res.n_selected], \
        (list(got["counts"]), res.n_candidates, res.n_selected)

"""GNMR oracle: plain, slow, double-precision CPU restatement of the per-step
GNMR monitor, used to check the CUDA path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference legs may import this package.  The
product path (``paper_2606_00539_gb300``) never imports it and shares no code
with it.

The arithmetic lives in ``gnmr_oracle.c`` (plain C, double precision, built by
:func:`build`); this module only marshals numpy arrays through ctypes.

* :func:`unit_norms` -- Eq. local_gradient: n_b = ||g_b||_2 (Sec. 2).
* :class:`Controller` -- Algorithm 1 (GNMR, Delta-GNMR, historical mean,
  window queue; Sec. 3.1-3.2) followed by Algorithm 2 (combined risk,
  candidate pool, Top_maxO, lock bookkeeping; Sec. 3.3).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gnmr_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle_gnmr.so")

DTYPE_F32 = 0
DTYPE_BF16 = 1

_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into ``oracle/liboracle_gnmr.so`` (plain -O2, no
    fast-math) and return its path."""
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-Wall", "-shared",
                               "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    P = ctypes.c_void_p
    lib.oracle_unit_norms.argtypes = [P, ctypes.c_int, P, P, ctypes.c_int32, P]
    lib.oracle_unit_norms.restype = ctypes.c_int
    lib.oracle_unit_norms_segmented.argtypes = [P, ctypes.c_int, P, P, P, ctypes.c_int64,
                                                ctypes.c_int32, P]
    lib.oracle_unit_norms_segmented.restype = ctypes.c_int
    lib.oracle_fq_round.argtypes = [ctypes.c_float, ctypes.c_int]
    lib.oracle_fq_round.restype = ctypes.c_float
    lib.oracle_fake_quant.argtypes = [P, P, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, ctypes.c_int]
    lib.oracle_fake_quant.restype = ctypes.c_int
    lib.oracle_ctl_create.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                      ctypes.c_int32, ctypes.c_int64, ctypes.c_double,
                                      ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                      ctypes.c_double, P]
    lib.oracle_ctl_create.restype = P
    lib.oracle_ctl_destroy.argtypes = [P]
    lib.oracle_ctl_destroy.restype = None
    lib.oracle_ctl_step.argtypes = [P, P, ctypes.c_double, ctypes.c_double,
                                    P, P, P, P, P, P]
    lib.oracle_ctl_step.restype = ctypes.c_int
    lib.oracle_ctl_set_policy.argtypes = [P, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64,
                                          ctypes.c_double]
    lib.oracle_ctl_set_policy.restype = ctypes.c_int
    lib.oracle_ctl_get_policy_state.argtypes = [P, P, P]
    lib.oracle_ctl_get_policy_state.restype = None
    lib.oracle_ctl_set_policy_state.argtypes = [P, P, P]
    lib.oracle_ctl_set_policy_state.restype = None
    lib.oracle_delta_mem.argtypes = [P, P, ctypes.c_int32]
    lib.oracle_delta_mem.restype = ctypes.c_double
    lib.oracle_ctl_get_state.argtypes = [P, P, P, P, P, P, P]
    lib.oracle_ctl_get_state.restype = None
    lib.oracle_ctl_set_state.argtypes = [P, P, P, P, P, P, ctypes.c_int64]
    lib.oracle_ctl_set_state.restype = None
    _lib = lib
    return lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _arena_dtype(arena: np.ndarray) -> int:
    if arena.dtype == np.float32:
        return DTYPE_F32
    if arena.dtype == np.uint16:          # raw bfloat16 bit patterns
        return DTYPE_BF16
    raise TypeError("arena must be float32 or uint16 (bfloat16 bits), got %s" % arena.dtype)


def unit_norms(arena: np.ndarray, offsets, lengths) -> np.ndarray:
    """n_b = ||g_b||_2 for every unit (Eq. local_gradient), summed
    sequentially in double.  ``arena`` is a flat float32 array or a flat
    uint16 array holding bfloat16 bit patterns; ``offsets``/``lengths`` are in
    elements."""
    arena = np.ascontiguousarray(arena).reshape(-1)
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    ln = np.ascontiguousarray(lengths, dtype=np.int64)
    if off.shape != ln.shape:
        raise ValueError("offsets and lengths differ in length")
    if len(off) and (np.any(off < 0) or np.any(ln < 0) or np.max(off + ln) > arena.size):
        raise ValueError("unit layout exceeds the arena")
    out = np.empty(len(off), dtype=np.float64)
    rc = _load().oracle_unit_norms(_ptr(arena), _arena_dtype(arena), _ptr(off), _ptr(ln),
                                   len(off), _ptr(out))
    if rc != 0:
        raise RuntimeError("oracle_unit_norms failed")
    return out


def unit_norms_threaded(arena: np.ndarray, offsets, lengths, threads: int) -> np.ndarray:
    """Same values as :func:`unit_norms`; units are split into contiguous
    groups of about equal element count and each group runs the same plain C
    loop on its own host thread (ctypes releases the GIL)."""
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    ln = np.ascontiguousarray(lengths, dtype=np.int64)
    U = len(off)
    threads = max(1, min(int(threads), U))
    if threads == 1:
        return unit_norms(arena, off, ln)
    cum = np.concatenate([[0], np.cumsum(ln)])
    cuts = np.searchsorted(cum, np.linspace(0, cum[-1], threads + 1)[1:-1])
    bounds = [0] + sorted(set(int(c) for c in cuts if 0 < c < U)) + [U]
    out = np.empty(U, dtype=np.float64)

    def run(i):
        a, b = bounds[i], bounds[i + 1]
        out[a:b] = unit_norms(arena, off[a:b], ln[a:b])

    with ThreadPoolExecutor(max_workers=len(bounds) - 1) as ex:
        list(ex.map(run, range(len(bounds) - 1)))
    return out


def unit_norms_segmented(arena: np.ndarray, offsets, lengths, segment_unit, num_units: int,
                         threads: int = 1) -> np.ndarray:
    """n_b over units made of several segments (Eq. local_gradient for a
    whole block, Sec. 3.4).  ``offsets``/``lengths``/``segment_unit`` describe
    the segments; the units are split over ``threads`` host threads, each
    running the same plain C loop over its units' segments."""
    arena = np.ascontiguousarray(arena).reshape(-1)
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    ln = np.ascontiguousarray(lengths, dtype=np.int64)
    su = np.ascontiguousarray(segment_unit, dtype=np.int32)
    if not (off.shape == ln.shape == su.shape):
        raise ValueError("segment arrays differ in length")
    if len(off) and (np.any(off < 0) or np.any(ln < 0) or np.max(off + ln) > arena.size
                     or su.min() < 0 or su.max() >= num_units):
        raise ValueError("segment layout exceeds the arena or the unit range")
    lib = _load()
    dt = _arena_dtype(arena)
    out = np.zeros(num_units, dtype=np.float64)
    threads = max(1, min(int(threads), num_units))
    bounds = np.linspace(0, num_units, threads + 1).astype(int)

    def run(i):
        a, b = bounds[i], bounds[i + 1]
        sel = np.nonzero((su >= a) & (su < b))[0]
        part = np.empty(b - a, dtype=np.float64)
        o = np.ascontiguousarray(off[sel])       # kept alive across the C call
        n = np.ascontiguousarray(ln[sel])
        u = np.ascontiguousarray(su[sel] - a, dtype=np.int32)
        rc = lib.oracle_unit_norms_segmented(_ptr(arena), dt, _ptr(o), _ptr(n), _ptr(u), len(sel),
                                             b - a, _ptr(part))
        if rc != 0:
            raise RuntimeError("oracle_unit_norms_segmented failed")
        out[a:b] = part

    if threads == 1:
        run(0)
    else:
        with ThreadPoolExecutor(max_workers=threads) as ex:
            list(ex.map(run, range(threads)))
    return out


POLICY_ACTIVE_CAP, POLICY_ADMISSION_CAP, POLICY_STATIC_TOP = 0, 1, 2

FQ_NONE, FQ_E2M1, FQ_E3M2, FQ_E4M3, FQ_E5M2 = 0, 1, 2, 3, 4


def delta_mem(mask, cost) -> float:
    """Eq. generic-memory-bound: the extra saved-activation memory of the
    units on the recovery path, Delta M_t = sum over b in A_t of c_b."""
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    c = np.ascontiguousarray(cost, dtype=np.float64)
    return float(_load().oracle_delta_mem(_ptr(m), _ptr(c), len(m)))


def fq_round(v: float, code: int) -> float:
    """Nearest value of minifloat format ``code`` to the fp32 value v."""
    return float(_load().oracle_fq_round(float(v), int(code)))


def fake_quant(x: np.ndarray, code: int) -> np.ndarray:
    """Per-token fake quantization (App. E.2) of a [rows, cols] float32 array
    or uint16 array of bfloat16 bits; returns a new array of the same kind."""
    x = np.ascontiguousarray(x)
    if x.ndim != 2:
        raise ValueError("x must be [rows, cols]")
    out = np.empty_like(x)
    rc = _load().oracle_fake_quant(_ptr(x), _ptr(out), _arena_dtype(x), x.shape[0], x.shape[1],
                                   int(code))
    if rc != 0:
        raise ValueError("bad format or dtype")
    return out


@dataclass
class StepResult:
    gnmr: np.ndarray      # GNMR_{b,t}
    dgnmr: np.ndarray     # Delta-GNMR_{b,t}
    risk: np.ndarray      # R_{b,t}
    mask: np.ndarray      # uint8, 1 = b in A_t (recovery path)
    lock: np.ndarray      # Lock_b after the step
    n_candidates: int     # |C_t|
    n_selected: int       # |A_t|


class Controller:
    """Per-unit state plus Algorithms 1 and 2, one call of :meth:`step` per
    training step.  ``alpha``/``beta`` are (init, main) pairs: the init value
    holds for steps t <= ``warmup_steps`` (two-stage schedule)."""

    def __init__(self, num_units: int, window: int, max_o: int, lock_len: int,
                 alpha=(1.5, 1.5), beta=(1.5, 1.5), warmup_steps: int = 0,
                 eps: float = 1e-8, recoverable=None, policy: int = 0,
                 forced_recovery_steps: int = 0, static_warmup_steps: int = 0,
                 static_fraction: float = 0.25):
        self.num_units = int(num_units)
        self.window = int(window)
        lib = _load()
        rec = None
        if recoverable is not None:
            rec = np.ascontiguousarray(recoverable, dtype=np.uint8)
            if rec.shape != (self.num_units,):
                raise ValueError("recoverable must have one flag per unit")
        self._h = lib.oracle_ctl_create(self.num_units, self.window, int(max_o), int(lock_len),
                                        int(warmup_steps), float(alpha[0]), float(alpha[1]),
                                        float(beta[0]), float(beta[1]), float(eps),
                                        None if rec is None else _ptr(rec))
        if not self._h:
            raise ValueError("invalid oracle controller configuration")
        if lib.oracle_ctl_set_policy(self._h, int(policy), int(forced_recovery_steps),
                                     int(static_warmup_steps), float(static_fraction)) != 0:
            raise ValueError("invalid oracle policy")

    def close(self):
        if getattr(self, "_h", None):
            _load().oracle_ctl_destroy(self._h)
            self._h = None

    def __del__(self):
        self.close()

    def step(self, norms, alpha: float = float("nan"), beta: float = float("nan")) -> StepResult:
        n = np.ascontiguousarray(norms, dtype=np.float64)
        if n.shape != (self.num_units,):
            raise ValueError("one norm per unit expected")
        U = self.num_units
        g, d, r = (np.empty(U, np.float64) for _ in range(3))
        mask = np.empty(U, np.uint8)
        lock = np.empty(U, np.int32)
        counts = np.empty(2, np.int32)
        _load().oracle_ctl_step(self._h, _ptr(n), float(alpha), float(beta), _ptr(g), _ptr(d),
                                _ptr(r), _ptr(mask), _ptr(lock), _ptr(counts))
        return StepResult(g, d, r, mask, lock, int(counts[0]), int(counts[1]))

    def get_state(self) -> dict:
        U, w = self.num_units, self.window
        st = dict(A=np.empty(U, np.float64), k=np.empty(U, np.int64),
                  Q=np.empty(U * w, np.float64), qlen=np.empty(U, np.int32),
                  lock=np.empty(U, np.int32))
        t = ctypes.c_int64(0)
        _load().oracle_ctl_get_state(self._h, _ptr(st["A"]), _ptr(st["k"]), _ptr(st["Q"]),
                                     _ptr(st["qlen"]), _ptr(st["lock"]), ctypes.byref(t))
        st["Q"] = st["Q"].reshape(U, w)
        st["t"] = int(t.value)
        return st

    def policy_state(self) -> dict:
        active = np.empty(self.num_units, np.uint8)
        gsum = np.empty(self.num_units, np.float64)
        _load().oracle_ctl_get_policy_state(self._h, _ptr(active), _ptr(gsum))
        return dict(active=active, gsum=gsum)

    def set_policy_state(self, st: dict) -> None:
        active = np.ascontiguousarray(st["active"], np.uint8)
        gsum = np.ascontiguousarray(st["gsum"], np.float64)
        _load().oracle_ctl_set_policy_state(self._h, _ptr(active), _ptr(gsum))

    def set_state(self, st: dict) -> None:
        A = np.ascontiguousarray(st["A"], np.float64)
        k = np.ascontiguousarray(st["k"], np.int64)
        Q = np.ascontiguousarray(st["Q"], np.float64).reshape(-1)
        qlen = np.ascontiguousarray(st["qlen"], np.int32)
        lock = np.ascontiguousarray(st["lock"], np.int32)
        _load().oracle_ctl_set_state(self._h, _ptr(A), _ptr(k), _ptr(Q), _ptr(qlen),
                                     _ptr(lock), int(st["t"]))

"""Seeded synthetic gradient workloads for the GNMR monitor.

Input generation only: unit layouts shaped like the paper's models, per-unit
per-step gradient scales (log-normal levels, a 1 %/step random walk, spikes,
ramps, unrouted MoE experts), and a GPU fill kernel (``tracegen.cu``) that
writes scale * N(0, 1) into each unit.  Nothing here computes a norm, a
ratio or a selection; both the CUDA path's tests and the oracle read the
arenas generated here.

Workloads (the model shapes follow Table 8 / Sec. 5.3 / the MoE appendix of the
paper; the trace statistics stand in for real training gradients, which need
datasets and checkpoints that are not used here):

1. ``tiny``        64 units, lengths log-uniform in [1K, 64K], fp32, 200 steps
2. ``llama2-1.3b`` 24 layers x 7 linears (168 units), bf16, 100 steps
3. ``llama2-13b``  40 layers x 7 linears (280 units, 12.69 G elements), bf16, 20 steps
4. ``moe``         27 layers x (4 attention + 64 routed x 3 + 2 shared x 3) = 5454 units,
                   bf16, 30 % of routed experts unrouted (exact zeros) per step, 50 steps
5. ``aq-stress``   100 000 units, lengths log-uniform in [256, 16K], fp32, 50 steps,
                   5 % spikes per step and a ramp family
"""
from __future__ import annotations

import ctypes
import math
import os
import shutil
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tracegen.cu")
LIB_PATH = os.path.join(_HERE, "libgnmr_tracegen.so")

NAMES = {1: "tiny", 2: "llama2-1.3b", 3: "llama2-13b", 4: "moe", 5: "aq-stress"}
IDS = {v: k for k, v in NAMES.items()}


@dataclass
class Workload:
    name: str
    dtype: str                      # "f32" or "bf16"
    offsets: np.ndarray             # int64 [S], elements, one per tensor (segment)
    lengths: np.ndarray             # int64 [S]
    recoverable: np.ndarray         # uint8 [U]
    arena_elems: int
    steps: int
    window: int
    max_o: int
    lock_len: int
    alpha: tuple
    beta: tuple
    warmup_steps: int
    eps: float
    seed: int
    scales: np.ndarray              # float64 [steps, S]; 0 = unrouted (exact zeros)
    kinds: list = field(default_factory=list)
    segment_unit: np.ndarray | None = None   # int32 [S]: unit of each tensor; None = one each
    group: str = "tensor"

    @property
    def num_segments(self) -> int:
        return len(self.offsets)

    @property
    def num_units(self) -> int:
        if self.segment_unit is None:
            return len(self.offsets)
        return int(self.segment_unit.max()) + 1

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    @property
    def grad_elems(self) -> int:
        return int(self.lengths.sum())

    @property
    def grad_bytes(self) -> int:
        return self.grad_elems * self.elem_bytes

    def monitor_kwargs(self) -> dict:
        kw = dict(dtype=self.dtype, recoverable=self.recoverable, window=self.window,
                  max_o=self.max_o, lock_len=self.lock_len, alpha=self.alpha, beta=self.beta,
                  warmup_steps=self.warmup_steps, eps=self.eps)
        if self.segment_unit is not None:
            kw.update(segment_unit=self.segment_unit, num_units=self.num_units)
        return kw

    def controller_kwargs(self) -> dict:
        return dict(window=self.window, max_o=self.max_o, lock_len=self.lock_len,
                    alpha=self.alpha, beta=self.beta, warmup_steps=self.warmup_steps,
                    eps=self.eps, recoverable=self.recoverable)


def _pack(lengths, elem_bytes):
    """Packed offsets, each unit starting on a 16-byte boundary."""
    align = 16 // elem_bytes
    off = np.zeros(len(lengths), np.int64)
    pos = 0
    for i, n in enumerate(lengths):
        off[i] = pos
        pos += int(n)
        pos = (pos + align - 1) // align * align
    return off, int(pos)


def _loguniform_int(rng, lo, hi, size):
    return np.round(np.exp(rng.uniform(math.log(lo), math.log(hi), size))).astype(np.int64)


def _drift_scales(rng, steps, U, sigma=0.01):
    s0 = np.exp(rng.standard_normal(U))                       # LogNormal(0, 1) level
    walk = np.cumsum(sigma * rng.standard_normal((steps, U)), axis=0)
    walk -= walk[0]
    return s0[None, :] * np.exp(walk)


def _spikes(rng, scales, count, lo, hi, max_len, first_step=2):
    steps, U = scales.shape
    for _ in range(count):
        u = int(rng.integers(0, U))
        t = int(rng.integers(first_step, steps))
        dur = int(rng.integers(1, max_len + 1))
        f = math.exp(rng.uniform(math.log(lo), math.log(hi)))
        scales[t:t + dur, u] *= f


def _linear_layout(layers, shapes, shrink):
    lens, kinds = [], []
    for layer in range(layers):
        for name, (r, c) in shapes:
            r2, c2 = max(1, -(-r // shrink)), max(1, -(-c // shrink))
            lens.append(r2 * c2)
            kinds.append(f"L{layer}.{name}")
    return np.array(lens, np.int64), kinds


def _grouping(cid, kinds, group):
    """segment -> unit map for block-level units (Sec. 3.4): ``block`` makes
    every transformer layer one unit; ``expert`` (MoE only) makes the attention
    projections of a layer one unit and every expert's three matrices one."""
    if group == "tensor":
        return None
    if cid not in (2, 3, 4):
        raise ValueError("block/expert grouping applies to the model layouts (configs 2-4)")
    keys = []
    for k in kinds:
        layer, name = k.split(".", 1)
        if group == "block":
            keys.append(layer)
        elif group == "expert" and cid == 4:
            keys.append(layer + "." + (name.split(".")[0] if "." in name else "attn"))
        else:
            raise ValueError(f"unknown grouping {group!r}")
    ids, seen = [], {}
    for key in keys:
        ids.append(seen.setdefault(key, len(seen)))
    return np.array(ids, np.int32)


def make(config, seed: int = 0, shrink: int = 1, steps: int | None = None,
         group: str = "tensor") -> Workload:
    """Builds workload ``config`` (1-5 or its name).  ``shrink`` divides every
    matrix dimension (configs 2-4) or unit length (configs 1, 5) to make a
    small case with the same structure; ``steps`` overrides the step count.
    ``group`` = "tensor" (one unit per weight tensor), "block" (one unit per
    transformer layer) or "expert" (MoE: attention and each expert grouped)."""
    cid = IDS.get(config, config)
    if cid not in NAMES:
        raise ValueError(f"unknown workload {config!r}")
    rng = np.random.default_rng([seed, cid])
    kinds: list = []
    if cid == 1:
        U, T = 64, 200
        lengths = np.maximum(1, _loguniform_int(rng, 1024, 65536, U) // shrink)
        dtype, window, max_o, lock_len = "f32", 8, 4, 5
        alpha, beta = (1.5, 1.1), (1.5, 1.5)
        T = steps or T
        scales = _drift_scales(rng, T, U)
        _spikes(rng, scales, 10, 10.0, 1000.0, 3)
        warm = math.ceil(0.025 * T)
    elif cid in (2, 3):
        d, f, L, T = (2048, 5504, 24, 100) if cid == 2 else (5120, 13824, 40, 20)
        shapes = [("q", (d, d)), ("k", (d, d)), ("v", (d, d)), ("o", (d, d)),
                  ("gate", (f, d)), ("up", (f, d)), ("down", (d, f))]
        lengths, kinds = _linear_layout(L, shapes, shrink)
        U = len(lengths)
        dtype = "bf16"
        window, max_o, lock_len = (8, 8, 10) if cid == 2 else (5, 16, 10)
        alpha, beta = (1.5, 1.1), (1.5, 1.5)
        T = steps or T
        scales = _drift_scales(rng, T, U)
        if cid == 2:
            _spikes(rng, scales, 20, 10.0, 1000.0, 3)
        else:
            for t in range(2, T):                               # 1-2 one-step spikes per step
                for _ in range(int(rng.integers(1, 3))):
                    u = int(rng.integers(0, U))
                    scales[t, u] *= math.exp(rng.uniform(math.log(10.0), math.log(1000.0)))
        warm = math.ceil(0.025 * T)
    elif cid == 4:
        d, fe, L, T, E, S = 2048, 1408, 27, 50, 64, 2
        attn = [("q", (d, d)), ("k", (d, d)), ("v", (d, d)), ("o", (d, d))]
        expert = [("gate", (fe, d)), ("up", (fe, d)), ("down", (d, fe))]
        shapes = list(attn)
        for e in range(E):
            shapes += [(f"e{e}.{n}", s) for n, s in expert]
        for e in range(S):
            shapes += [(f"shared{e}.{n}", s) for n, s in expert]
        lengths, kinds = _linear_layout(L, shapes, shrink)
        U = len(lengths)
        dtype, window, max_o, lock_len = "bf16", 8, 32, 8
        alpha, beta = (1.5, 1.1), (1.5, 1.5)
        T = steps or T
        scales = _drift_scales(rng, T, U)
        _spikes(rng, scales, 20, 10.0, 1000.0, 3)
        per_layer = len(shapes)
        unrouted = rng.random((T, L, E)) < 0.3                  # Bernoulli(0.3) per expert
        for layer in range(L):
            for e in range(E):
                cols = [layer * per_layer + 4 + 3 * e + j for j in range(3)]
                for c in cols:
                    scales[unrouted[:, layer, e], c] = 0.0
        warm = math.ceil(0.025 * T)
    else:
        U, T = 100_000, 50
        lengths = np.maximum(1, _loguniform_int(rng, 256, 16384, U) // shrink)
        dtype, window, max_o, lock_len = "f32", 8, 64, 3
        alpha, beta = (1.5, 1.5), (1.3, 1.3)
        T = steps or T
        scales = _drift_scales(rng, T, U)
        spike = rng.random((T, U)) < 0.05
        factor = np.exp(rng.uniform(math.log(4.0), math.log(1e4), (T, U)))
        spike[:2] = False
        scales = np.where(spike, scales * factor, scales)
        ramp_units = rng.choice(U, size=U // 100, replace=False)
        for u in ramp_units:                                    # abrupt jump, then x1.1 per step
            onset = int(rng.integers(window + 1, 31))
            c0 = math.exp(rng.uniform(math.log(1.5), math.log(3.0)))
            for k in range(20):
                if onset + k < T:
                    scales[onset + k, u] *= c0 * (1.1 ** k)
        warm = 0
    esize = 2 if dtype == "bf16" else 4
    offsets, arena_elems = _pack(lengths, esize)
    seg_unit = _grouping(cid, kinds, group)
    U = len(lengths) if seg_unit is None else int(seg_unit.max()) + 1
    if seg_unit is not None:
        max_o = max(1, min(max_o, U // 4))       # the budget scales with the coarser units
    return Workload(name=NAMES[cid] + ("" if group == "tensor" else f"/{group}"), dtype=dtype,
                    offsets=offsets, lengths=lengths, recoverable=np.ones(U, np.uint8),
                    arena_elems=arena_elems, steps=T, window=window, max_o=max_o,
                    lock_len=lock_len, alpha=alpha, beta=beta, warmup_steps=warm, eps=1e-8,
                    seed=seed, scales=np.ascontiguousarray(scales), kinds=kinds,
                    segment_unit=seg_unit, group=group)


def redraw_factor(seed: int, unit: int, step: int, attempt: int) -> float:
    """Scale multiplier within +-1 % used to move a unit away from a decision
    boundary, keyed by (seed, unit, step, attempt)."""
    r = np.random.default_rng([seed, unit, step, attempt, 7919])
    return float(math.exp(r.uniform(-0.01, 0.01)))


# ---------------------------------------------------------------------------
# GPU fill (tracegen.cu)
# ---------------------------------------------------------------------------

def build(force: bool = False) -> str:
    stale = (not os.path.exists(LIB_PATH)
             or os.path.getmtime(LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
        tmp = LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3",
                               "-std=c++17", "-Xcompiler", "-fPIC", "-shared", "-cudart", "static",
                               "-o", tmp, _SRC])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} missing: run workloads.build()")
        lib = ctypes.CDLL(LIB_PATH)
        P = ctypes.c_void_p
        lib.tracegen_fill.argtypes = [P, ctypes.c_int, P, P, P, ctypes.c_int64, P, P, P,
                                      ctypes.c_uint32, ctypes.c_uint32, P]
        lib.tracegen_fill.restype = ctypes.c_int
        _lib = lib
    return _lib


class Filler:
    """Writes workload gradients into a device arena with the Philox fill
    kernel, one weight tensor (segment) at a time.  One instance per
    (workload, device)."""

    CHUNK = 1 << 20

    def __init__(self, w: Workload, device):
        import torch
        self.torch = torch
        self.w = w
        self.device = torch.device(device)
        self._off = torch.from_numpy(w.offsets).to(self.device)
        self._scale = torch.zeros(w.num_segments, dtype=torch.float64, device=self.device)
        self._attempt = torch.zeros(w.num_segments, dtype=torch.int32, device=self.device)
        self._all_tasks = self._tasks(np.arange(w.num_segments))

    def _tasks(self, units):
        torch = self.torch
        tu, ts, tc = [], [], []
        for u in units:
            n = int(self.w.lengths[u])
            for s in range(0, n, self.CHUNK):
                tu.append(u)
                ts.append(s)
                tc.append(min(self.CHUNK, n - s))
        mk = lambda a: torch.tensor(np.array(a, np.int64), device=self.device)
        return mk(tu), mk(ts), mk(tc), len(tu)

    def new_arena(self, fill_value=float("nan")):
        torch = self.torch
        dt = torch.bfloat16 if self.w.dtype == "bf16" else torch.float32
        return torch.full((self.w.arena_elems,), fill_value, dtype=dt, device=self.device)

    def fill(self, arena, step: int, scales=None, attempts=None, units=None, stream=None):
        """Writes step ``step`` of every segment (or of the segments listed in
        ``units``) into arena.  ``scales``/``attempts`` (per segment) default
        to the workload's scales and 0."""
        torch = self.torch
        sc = self.w.scales[step] if scales is None else scales
        self._scale.copy_(torch.from_numpy(np.ascontiguousarray(sc, np.float64)))
        at = np.zeros(self.w.num_segments, np.int32) if attempts is None else attempts
        self._attempt.copy_(torch.from_numpy(np.ascontiguousarray(at, np.int32)))
        tu, ts, tc, n = self._all_tasks if units is None else self._tasks(units)
        st = stream.cuda_stream if stream is not None else torch.cuda.current_stream(self.device).cuda_stream
        rc = _load().tracegen_fill(arena.data_ptr(), 1 if self.w.dtype == "bf16" else 0,
                                   tu.data_ptr(), ts.data_ptr(), tc.data_ptr(), n,
                                   self._off.data_ptr(), self._scale.data_ptr(),
                                   self._attempt.data_ptr(), self.w.seed & 0xffffffff, step, st)
        if rc != 0:
            raise RuntimeError(f"tracegen_fill failed with CUDA error {rc}")

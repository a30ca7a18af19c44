"""torch-facing wrapper of the GNMR C ABI.  PyTorch supplies device memory and
the CUDA stream; every step of the monitor runs in libgnmr's kernel."""
from __future__ import annotations

import ctypes
import math

import numpy as np

from . import _native as N

_DTYPES = {"f32": N.GNMR_DTYPE_F32, "float32": N.GNMR_DTYPE_F32,
           "bf16": N.GNMR_DTYPE_BF16, "bfloat16": N.GNMR_DTYPE_BF16}
_LOOP_SHAPES = {"auto": N.GNMR_LOOP_AUTO, "small": N.GNMR_LOOP_SMALL_UNITS,
                "large": N.GNMR_LOOP_LARGE_UNITS}


def _torch():
    import torch
    return torch


class Monitor:
    """The GNMR per-step monitor for one flat gradient arena.

    offsets, lengths: element offset and length in the arena of every unit,
    or of every segment when segment_unit is given (segment_unit[s] = the
    unit of segment s, for units that span several tensors, e.g. a whole
    transformer block; num_units defaults to max(segment_unit) + 1).
    recoverable: per-unit flags (B_rec); None = every unit recoverable.
    alpha, beta: (init, main) thresholds; the init values hold for steps
    t <= warmup_steps (two-stage schedule).  A scalar means both stages.
    policy, forced_recovery_steps, static_warmup_steps, static_fraction: the
    recovery policy variants of include/gnmr.h; unit_cost: per-unit c_b for
    the Delta M_t statistic.  loop_shape: "auto", "small" or "large", the
    kernel's streaming-loop shape (norms agree within rounding across shapes).
    """

    def __init__(self, offsets, lengths, *, dtype="bf16", recoverable=None, window=8, max_o=4,
                 lock_len=1, alpha=(1.5, 1.1), beta=(1.5, 1.5), warmup_steps=0, eps=1e-8,
                 device=0, segment_unit=None, num_units=None, policy=0, forced_recovery_steps=0,
                 static_warmup_steps=0, static_fraction=0.25, unit_cost=None, loop_shape="auto"):
        self._h = None
        off = np.ascontiguousarray(offsets, dtype=np.int64)
        ln = np.ascontiguousarray(lengths, dtype=np.int64)
        if off.ndim != 1 or off.shape != ln.shape:
            raise ValueError("offsets and lengths must be 1-D arrays of equal length")
        seg = None
        if segment_unit is not None:
            seg = np.ascontiguousarray(segment_unit, dtype=np.int32)
            if seg.shape != off.shape:
                raise ValueError("segment_unit must have one entry per segment")
            if num_units is None:
                num_units = int(seg.max()) + 1 if len(seg) else 0
        elif num_units is not None and num_units != len(off):
            raise ValueError("num_units without segment_unit must equal len(offsets)")
        U = len(off) if num_units is None else int(num_units)
        rec = None
        if recoverable is not None:
            rec = np.ascontiguousarray(recoverable, dtype=np.uint8)
            if rec.shape != (U,):
                raise ValueError("recoverable must have one flag per unit")
        if isinstance(alpha, (int, float)):
            alpha = (alpha, alpha)
        if isinstance(beta, (int, float)):
            beta = (beta, beta)
        if dtype not in _DTYPES:
            raise ValueError(f"dtype must be one of {sorted(_DTYPES)}")
        cfg = N.gnmr_config_defaults()
        cfg.num_units = U
        if seg is not None:
            cfg.num_segments = len(seg)
            cfg.segment_unit = seg.ctypes.data
        cfg.offsets = off.ctypes.data
        cfg.lengths = ln.ctypes.data
        cfg.recoverable = None if rec is None else rec.ctypes.data
        cfg.dtype = _DTYPES[dtype]
        cfg.window = int(window)
        cfg.max_o = int(max_o)
        cfg.lock_len = int(lock_len)
        cfg.alpha_init, cfg.alpha_main = float(alpha[0]), float(alpha[1])
        cfg.beta_init, cfg.beta_main = float(beta[0]), float(beta[1])
        cfg.warmup_steps = int(warmup_steps)
        cfg.eps = float(eps)
        cfg.device = int(device.index if hasattr(device, "index") else device)
        cfg.policy = int(policy)
        cfg.forced_recovery_steps = int(forced_recovery_steps)
        cfg.static_warmup_steps = int(static_warmup_steps)
        cfg.static_fraction = float(static_fraction)
        if loop_shape not in _LOOP_SHAPES:
            raise ValueError(f"loop_shape must be one of {sorted(_LOOP_SHAPES)}")
        cfg.loop_shape = _LOOP_SHAPES[loop_shape]
        cost = None
        if unit_cost is not None:
            cost = np.ascontiguousarray(unit_cost, dtype=np.float64)
            if cost.shape != (U,):
                raise ValueError("unit_cost must have one entry per unit")
            cfg.unit_cost = cost.ctypes.data
        self._h = N.gnmr_create(cfg)
        self.num_units = U
        self.dtype = cfg.dtype
        self.device_index = cfg.device
        self.arena_elems_min = int(self.info()["arena_elems_min"])

    # -- lifetime -----------------------------------------------------------
    def close(self) -> None:
        if self._h:
            N.gnmr_destroy(self._h)
            self._h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- queries ------------------------------------------------------------
    def info(self) -> dict:
        return N.gnmr_get_info(self._h)

    def set_thresholds(self, alpha: float = math.nan, beta: float = math.nan) -> None:
        N.gnmr_set_thresholds(self._h, alpha, beta)

    # -- the step -----------------------------------------------------------
    def new_stats(self) -> dict:
        torch = _torch()
        dev = torch.device("cuda", self.device_index)
        U = self.num_units
        return {
            "norm": torch.empty(U, dtype=torch.float64, device=dev),
            "gnmr": torch.empty(U, dtype=torch.float64, device=dev),
            "dgnmr": torch.empty(U, dtype=torch.float64, device=dev),
            "risk": torch.empty(U, dtype=torch.float64, device=dev),
            "lock": torch.empty(U, dtype=torch.int32, device=dev),
            "counts": torch.empty(2, dtype=torch.int32, device=dev),
            "delta_mem": torch.zeros(1, dtype=torch.float64, device=dev),
        }

    def _check_tensor(self, t, name, dtype, numel=None):
        torch = _torch()
        if not isinstance(t, torch.Tensor) or not t.is_cuda or t.device.index != self.device_index:
            raise ValueError(f"{name} must be a CUDA tensor on device {self.device_index}")
        if t.dtype != dtype:
            raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if numel is not None and t.numel() < numel:
            raise ValueError(f"{name} must hold at least {numel} elements")

    def _stats_struct(self, stats):
        torch = _torch()
        if stats is None:
            return None
        st = N.gnmr_stats()
        for key, dt, n in (("norm", torch.float64, self.num_units),
                           ("gnmr", torch.float64, self.num_units),
                           ("dgnmr", torch.float64, self.num_units),
                           ("risk", torch.float64, self.num_units),
                           ("lock", torch.int32, self.num_units),
                           ("counts", torch.int32, 2),
                           ("delta_mem", torch.float64, 1)):
            if stats.get(key) is not None:
                self._check_tensor(stats[key], key, dt, n)
                setattr(st, key, stats[key].data_ptr())
        return st

    def _stream_handle(self, stream, device):
        torch = _torch()
        if stream is None:
            stream = torch.cuda.current_stream(device)
        return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)

    def prepare_step(self, arena, mask=None, stats: dict | None = None, stream=None):
        """Validates and marshals step()'s arguments once and returns a
        callable that enqueues one step with them: each call is one C call
        (for loops where the Python cost of step() would gap the GPU).  The
        tensors' storage and the stream are fixed at preparation; their
        contents may change between calls (e.g. the next step's gradients
        written into the same arena).  The callable returns the mask."""
        torch = _torch()
        dev = self._check_arena(arena)
        if mask is None:
            mask = torch.empty(self.num_units, dtype=torch.uint8, device=dev)
        self._check_tensor(mask, "mask", torch.uint8, self.num_units)
        st = self._stats_struct(stats)
        fn = N.load().gnmr_step
        args = (self._h, arena.data_ptr(), int(arena.numel()), self._stream_handle(stream, dev),
                mask.data_ptr(), ctypes.byref(st) if st is not None else None)
        keep = (arena, mask, stats, st)            # storage the prepared call points into
        handle = self._h

        def run():
            if self._h != handle:
                raise ValueError("the monitor was closed")
            status = fn(*args)
            if status:
                N._check(status, handle)
            return keep[1]

        return run

    def step_partials(self, arena, sumsq=None, stream=None):
        """First half of a sharded step: per-unit sums of squares of this
        rank's local arena (fp64 tensor [U]); no controller state changes."""
        torch = _torch()
        dev = self._check_arena(arena)
        if sumsq is None:
            sumsq = torch.empty(self.num_units, dtype=torch.float64, device=dev)
        self._check_tensor(sumsq, "sumsq", torch.float64, self.num_units)
        N.gnmr_step_partials(self._h, arena.data_ptr(), arena.numel(),
                             self._stream_handle(stream, dev), sumsq.data_ptr())
        return sumsq

    def finish(self, sumsq, mask=None, stats: dict | None = None, stream=None):
        """Second half: one controller step on summed sums of squares."""
        torch = _torch()
        self._check_tensor(sumsq, "sumsq", torch.float64, self.num_units)
        if mask is None:
            mask = torch.empty(self.num_units, dtype=torch.uint8, device=sumsq.device)
        self._check_tensor(mask, "mask", torch.uint8, self.num_units)
        N.gnmr_finish(self._h, sumsq.data_ptr(), self._stream_handle(stream, sumsq.device),
                      mask.data_ptr(), self._stats_struct(stats))
        return mask

    def get_state(self, stream=None) -> bytes:
        """Checkpoint blob of the controller state (waits for the stream)."""
        torch = _torch()
        return N.gnmr_get_state(self._h, self._stream_handle(stream, torch.device("cuda", self.device_index)))

    def set_state(self, blob: bytes, stream=None) -> None:
        torch = _torch()
        N.gnmr_set_state(self._h, blob, self._stream_handle(stream, torch.device("cuda", self.device_index)))

    def _check_arena(self, arena):
        """The arena: a CUDA tensor on the handle's device, or a pinned CPU
        tensor, which the kernel reads in place over the host link."""
        torch = _torch()
        want = torch.bfloat16 if self.dtype == N.GNMR_DTYPE_BF16 else torch.float32
        if isinstance(arena, torch.Tensor) and not arena.is_cuda:
            if not arena.is_pinned():
                raise ValueError("a host arena must be pinned (pin_memory=True)")
            if arena.dtype != want:
                raise ValueError(f"arena must be {want}, got {arena.dtype}")
            if not arena.is_contiguous():
                raise ValueError("arena must be contiguous")
        else:
            self._check_tensor(arena, "arena", want)
        return torch.device("cuda", self.device_index)

    def step(self, arena, mask=None, stats: dict | None = None, stream=None):
        """Enqueues one GNMR step on `stream` (default: torch's current
        stream) and returns the uint8 mask tensor (1 = recovery path).
        `arena` is a CUDA tensor or a pinned CPU tensor (read in place)."""
        torch = _torch()
        dev = self._check_arena(arena)
        if mask is None:
            mask = torch.empty(self.num_units, dtype=torch.uint8, device=dev)
        self._check_tensor(mask, "mask", torch.uint8, self.num_units)
        N.gnmr_step(self._h, arena.data_ptr(), arena.numel(), self._stream_handle(stream, dev),
                    mask.data_ptr(), self._stats_struct(stats))
        return mask

"""torch-facing wrapper of the GNMR C ABI.  PyTorch supplies device memory and
the CUDA stream; every step of the monitor runs in libgnmr's kernel."""
from __future__ import annotations

import ctypes
import math

import numpy as np

from . import _native as N

_DTYPES = {"f32": N.GNMR_DTYPE_F32, "float32": N.GNMR_DTYPE_F32,
           "bf16": N.GNMR_DTYPE_BF16, "bfloat16": N.GNMR_DTYPE_BF16}


def _torch():
    import torch
    return torch


class Monitor:
    """The GNMR per-step monitor for one flat gradient arena.

    offsets, lengths: per-unit element offset and length in the arena.
    recoverable: per-unit flags (B_rec); None = every unit recoverable.
    alpha, beta: (init, main) thresholds; the init values hold for steps
    t <= warmup_steps (two-stage schedule).  A scalar means both stages.
    """

    def __init__(self, offsets, lengths, *, dtype="bf16", recoverable=None, window=8, max_o=4,
                 lock_len=1, alpha=(1.5, 1.1), beta=(1.5, 1.5), warmup_steps=0, eps=1e-8,
                 device=0):
        self._h = None
        off = np.ascontiguousarray(offsets, dtype=np.int64)
        ln = np.ascontiguousarray(lengths, dtype=np.int64)
        if off.ndim != 1 or off.shape != ln.shape:
            raise ValueError("offsets and lengths must be 1-D arrays of equal length")
        rec = None
        if recoverable is not None:
            rec = np.ascontiguousarray(recoverable, dtype=np.uint8)
            if rec.shape != off.shape:
                raise ValueError("recoverable must have one flag per unit")
        if isinstance(alpha, (int, float)):
            alpha = (alpha, alpha)
        if isinstance(beta, (int, float)):
            beta = (beta, beta)
        if dtype not in _DTYPES:
            raise ValueError(f"dtype must be one of {sorted(_DTYPES)}")
        cfg = N.gnmr_config_defaults()
        cfg.num_units = len(off)
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
        self._h = N.gnmr_create(cfg)
        self.num_units = len(off)
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

    def step(self, arena, mask=None, stats: dict | None = None, stream=None):
        """Enqueues one GNMR step on `stream` (default: torch's current
        stream) and returns the uint8 mask tensor (1 = recovery path)."""
        torch = _torch()
        want = torch.bfloat16 if self.dtype == N.GNMR_DTYPE_BF16 else torch.float32
        self._check_tensor(arena, "arena", want)
        if mask is None:
            mask = torch.empty(self.num_units, dtype=torch.uint8, device=arena.device)
        self._check_tensor(mask, "mask", torch.uint8, self.num_units)
        st = None
        if stats is not None:
            st = N.gnmr_stats()
            for key, dt, n in (("norm", torch.float64, self.num_units),
                               ("gnmr", torch.float64, self.num_units),
                               ("dgnmr", torch.float64, self.num_units),
                               ("risk", torch.float64, self.num_units),
                               ("lock", torch.int32, self.num_units),
                               ("counts", torch.int32, 2)):
                if stats.get(key) is not None:
                    self._check_tensor(stats[key], key, dt, n)
                    setattr(st, key, stats[key].data_ptr())
        if stream is None:
            stream = torch.cuda.current_stream(arena.device)
        s = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
        N.gnmr_step(self._h, arena.data_ptr(), arena.numel(), s, mask.data_ptr(), st)
        return mask

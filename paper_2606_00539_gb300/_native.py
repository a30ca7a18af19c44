"""ctypes binding of libgnmr (include/gnmr.h): the same entry points under the
same names, argument marshalling only.  Every step of the GNMR path runs in
the CUDA library; there is no Python or CPU fallback.  If the library has not
been built, :func:`load` raises.
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libgnmr.so")

GNMR_OK = 0
GNMR_ERR_INVALID_ARG = 1
GNMR_ERR_LAYOUT = 2
GNMR_ERR_CUDA = 3
GNMR_ERR_OOM = 4
GNMR_ERR_STATE = 5

GNMR_DTYPE_F32 = 0
GNMR_DTYPE_BF16 = 1

GNMR_FQ_NONE, GNMR_FQ_E2M1, GNMR_FQ_E3M2, GNMR_FQ_E4M3, GNMR_FQ_E5M2 = 0, 1, 2, 3, 4

GNMR_POLICY_ACTIVE_CAP, GNMR_POLICY_ADMISSION_CAP, GNMR_POLICY_STATIC_TOP = 0, 1, 2
GNMR_LOOP_AUTO, GNMR_LOOP_SMALL_UNITS, GNMR_LOOP_LARGE_UNITS = 0, 1, 2

_P = ctypes.c_void_p


class gnmr_config(ctypes.Structure):
    _fields_ = [
        ("num_units", ctypes.c_int32),
        ("offsets", _P),
        ("lengths", _P),
        ("recoverable", _P),
        ("dtype", ctypes.c_int32),
        ("window", ctypes.c_int32),
        ("max_o", ctypes.c_int32),
        ("lock_len", ctypes.c_int32),
        ("alpha_init", ctypes.c_double),
        ("alpha_main", ctypes.c_double),
        ("beta_init", ctypes.c_double),
        ("beta_main", ctypes.c_double),
        ("warmup_steps", ctypes.c_int64),
        ("eps", ctypes.c_double),
        ("device", ctypes.c_int32),
        ("num_segments", ctypes.c_int32),
        ("segment_unit", _P),
        ("policy", ctypes.c_int32),
        ("forced_recovery_steps", ctypes.c_int64),
        ("static_warmup_steps", ctypes.c_int64),
        ("static_fraction", ctypes.c_double),
        ("unit_cost", _P),
        ("loop_shape", ctypes.c_int32),
    ]


class gnmr_stats(ctypes.Structure):
    _fields_ = [
        ("norm", _P),
        ("gnmr", _P),
        ("dgnmr", _P),
        ("risk", _P),
        ("lock", _P),
        ("counts", _P),
        ("delta_mem", _P),
    ]


class gnmr_info(ctypes.Structure):
    _fields_ = [
        ("num_units", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("device", ctypes.c_int32),
        ("num_ctas", ctypes.c_int32),
        ("threads_per_cta", ctypes.c_int32),
        ("num_warps", ctypes.c_int32),
        ("num_partials", ctypes.c_int64),
        ("device_bytes", ctypes.c_int64),
        ("arena_elems_min", ctypes.c_int64),
        ("steps", ctypes.c_int64),
        ("loop_shape", ctypes.c_int32),
        ("num_runs", ctypes.c_int32),
    ]


class GnmrError(RuntimeError):
    def __init__(self, status: int, detail: str):
        super().__init__(f"{status_string(status)} ({detail})" if detail else status_string(status))
        self.status = status
        self.detail = detail


# name -> (restype, argtypes), one entry per function declared in gnmr.h
PROTOTYPES = {
    "gnmr_config_defaults": (None, [ctypes.POINTER(gnmr_config)]),
    "gnmr_create": (ctypes.c_int, [ctypes.POINTER(gnmr_config), ctypes.POINTER(_P)]),
    "gnmr_step": (ctypes.c_int, [_P, _P, ctypes.c_int64, _P, _P, ctypes.POINTER(gnmr_stats)]),
    "gnmr_set_thresholds": (ctypes.c_int, [_P, ctypes.c_double, ctypes.c_double]),
    "gnmr_get_info": (ctypes.c_int, [_P, ctypes.POINTER(gnmr_info)]),
    "gnmr_destroy": (ctypes.c_int, [_P]),
    "gnmr_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "gnmr_last_error": (ctypes.c_char_p, [_P]),
    "gnmr_plan_partition": (ctypes.c_int, [ctypes.c_int32, _P, ctypes.c_int32, ctypes.c_int32,
                                           _P, _P, _P, _P, _P]),
    "gnmr_unit_norms_static": (ctypes.c_int, [_P, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                              _P, _P, _P, _P]),
    "gnmr_actuator_create": (ctypes.c_int, [ctypes.c_int32, _P, _P, _P, ctypes.c_int32, ctypes.c_int32,
                                            ctypes.POINTER(_P)]),
    "gnmr_actuator_apply": (ctypes.c_int, [_P, _P, _P, ctypes.c_int64, _P, ctypes.c_int32, ctypes.c_int32,
                                           _P]),
    "gnmr_actuator_destroy": (ctypes.c_int, [_P]),
    "gnmr_step_partials": (ctypes.c_int, [_P, _P, ctypes.c_int64, _P, _P]),
    "gnmr_finish": (ctypes.c_int, [_P, _P, _P, _P, ctypes.POINTER(gnmr_stats)]),
    "gnmr_get_state": (ctypes.c_int, [_P, _P, _P, ctypes.c_int64, ctypes.POINTER(ctypes.c_int64)]),
    "gnmr_set_state": (ctypes.c_int, [_P, _P, _P, ctypes.c_int64]),
}

_lib = None


def load() -> ctypes.CDLL:
    """Loads the in-tree libgnmr.so.  Raises RuntimeError if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            f"{LIB_PATH} is missing: the GNMR CUDA library has not been built "
            "(python -m paper_2606_00539_gb300.build)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in PROTOTYPES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().gnmr_status_string(int(status)).decode()


def last_error(handle) -> str:
    return (load().gnmr_last_error(handle) or b"").decode()


def _check(status: int, handle=None) -> None:
    if status != GNMR_OK:
        raise GnmrError(status, last_error(handle))


def gnmr_config_defaults() -> gnmr_config:
    cfg = gnmr_config()
    load().gnmr_config_defaults(ctypes.byref(cfg))
    return cfg


def gnmr_create(cfg: gnmr_config) -> int:
    """Returns the handle (an opaque pointer value).  Raises GnmrError."""
    h = _P()
    st = load().gnmr_create(ctypes.byref(cfg), ctypes.byref(h))
    _check(st, None)
    return h.value


def gnmr_step(handle: int, d_arena: int, arena_elems: int, stream: int, d_mask: int,
              stats: gnmr_stats | None = None) -> None:
    st = load().gnmr_step(handle, d_arena, int(arena_elems), stream, d_mask,
                          ctypes.byref(stats) if stats is not None else None)
    _check(st, handle)


def gnmr_step_partials(handle: int, d_arena: int, arena_elems: int, stream: int, d_sumsq: int) -> None:
    _check(load().gnmr_step_partials(handle, d_arena, int(arena_elems), stream, d_sumsq), handle)


def gnmr_finish(handle: int, d_sumsq: int, stream: int, d_mask: int,
                stats: gnmr_stats | None = None) -> None:
    st = load().gnmr_finish(handle, d_sumsq, stream, d_mask,
                            ctypes.byref(stats) if stats is not None else None)
    _check(st, handle)


def gnmr_get_state(handle: int, stream: int = 0) -> bytes:
    """Returns the controller state blob."""
    lib = load()
    size = ctypes.c_int64(0)
    _check(lib.gnmr_get_state(handle, stream, None, 0, ctypes.byref(size)), handle)
    buf = ctypes.create_string_buffer(size.value)
    _check(lib.gnmr_get_state(handle, stream, buf, size.value, ctypes.byref(size)), handle)
    return buf.raw


def gnmr_set_state(handle: int, blob: bytes, stream: int = 0) -> None:
    buf = ctypes.create_string_buffer(bytes(blob), len(blob))
    _check(load().gnmr_set_state(handle, stream, buf, len(blob)), handle)


def gnmr_set_thresholds(handle: int, alpha: float, beta: float) -> None:
    _check(load().gnmr_set_thresholds(handle, float(alpha), float(beta)), handle)


def gnmr_get_info(handle: int) -> dict:
    info = gnmr_info()
    _check(load().gnmr_get_info(handle, ctypes.byref(info)), handle)
    return {name: getattr(info, name) for name, _ in gnmr_info._fields_}


def gnmr_destroy(handle: int) -> None:
    _check(load().gnmr_destroy(handle), None)


def gnmr_plan_partition(lengths, dtype: int, max_warps: int):
    """Host-only plan query; returns (run_unit, run_pos, first_warp, num_parts)
    as numpy arrays."""
    import numpy as np
    ln = np.ascontiguousarray(lengths, dtype=np.int64)
    U = len(ln)
    run_unit = np.zeros(max_warps + 1, np.int32)
    run_pos = np.zeros(max_warps + 1, np.int64)
    first = np.zeros(U, np.int32)
    parts = np.zeros(U, np.int32)
    nw = ctypes.c_int32(0)
    st = load().gnmr_plan_partition(U, ln.ctypes.data, int(dtype), int(max_warps),
                                    ctypes.addressof(nw), run_unit.ctypes.data,
                                    run_pos.ctypes.data, first.ctypes.data, parts.ctypes.data)
    _check(st, None)
    n = nw.value
    return run_unit[:n + 1], run_pos[:n + 1], first, parts


def gnmr_actuator_create(offsets, rows, cols, dtype: int, device: int = 0) -> int:
    import numpy as np
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    r = np.ascontiguousarray(rows, dtype=np.int64)
    c = np.ascontiguousarray(cols, dtype=np.int64)
    h = _P()
    st = load().gnmr_actuator_create(len(off), off.ctypes.data, r.ctypes.data, c.ctypes.data,
                                     int(dtype), int(device), ctypes.byref(h))
    _check(st, None)
    return h.value


def gnmr_actuator_apply(handle: int, d_in: int, d_out: int, arena_elems: int, d_mask,
                        lowcost_format: int, recovery_format: int, stream: int = 0) -> None:
    st = load().gnmr_actuator_apply(handle, d_in, d_out, int(arena_elems), d_mask,
                                    int(lowcost_format), int(recovery_format), stream)
    _check(st, None)


def gnmr_actuator_destroy(handle: int) -> None:
    _check(load().gnmr_actuator_destroy(handle), None)

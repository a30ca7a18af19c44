"""GB300-native GNMR per-step monitor (sm_103a).

The monitor reduces every unit's gradient to its L2 norm, updates the unit's
historical mean and GNMR window, forms GNMR and Delta-GNMR, and selects at
most maxO units for the recovery path under the lock interval -- one CUDA
kernel launch per training step, behind the C ABI in ``include/gnmr.h``.

* :mod:`._native` -- ctypes binding with the C entry points' names.
* :class:`Monitor` -- torch-facing wrapper (torch supplies memory and streams).
* :mod:`.build` -- compiles ``libgnmr.so`` for sm_103a.
"""
from ._native import GnmrError, load  # noqa: F401
from .monitor import Monitor  # noqa: F401

__all__ = ["Monitor", "GnmrError", "load"]

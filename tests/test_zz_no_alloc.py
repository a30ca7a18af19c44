"""gnmr_unit_norms_static: per-unit norms for callers that cannot allocate
device memory (a framework's caching allocator owns the GPU, a hook runs in
the middle of a step where cudaMalloc's device synchronisation would stall
it, or the deployment fixes its footprint up front).  Its scratch is a static
device array inside libgnmr, so it needs no handle.

Called through the C ABI and checked against gnmr_step's own norm output
(stats->norm) and against the oracle on the same bytes, twice in a row,
within the tolerance of the other parity tests.  Kept in its own file,
collected last."""
import numpy as np
import pytest

import workloads
from paper_2606_00539_gb300 import Monitor
from paper_2606_00539_gb300 import _native as N

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def _static_norms(lib, arena, w, out, stream=0):
    off = np.ascontiguousarray(w.offsets, np.int64)
    ln = np.ascontiguousarray(w.lengths, np.int64)
    dt = N.GNMR_DTYPE_BF16 if w.dtype == "bf16" else N.GNMR_DTYPE_F32
    return lib.gnmr_unit_norms_static(arena.data_ptr(), arena.numel(), dt, w.num_units,
                                      off.ctypes.data, ln.ctypes.data, out.data_ptr(), stream)


@pytest.mark.parametrize("config,shrink", [("llama2-13b", 16), ("aq-stress", 4), ("tiny", 1),
                                           ("llama2-13b", 1), ("aq-stress", 1)])
def test_static_norms_match_gnmr_step(config, shrink, cuda_device):
    import torch
    lib = N.load()
    import oracle
    w = workloads.make(config, shrink=shrink, steps=3)
    filler = workloads.Filler(w, cuda_device)
    arena = filler.new_arena()
    host = torch.empty(arena.numel(), dtype=arena.dtype, pin_memory=True)
    mon = Monitor(w.offsets, w.lengths, device=0, **w.monitor_kwargs())
    stats = mon.new_stats()
    try:
        for t in range(2):                      # two calls in a row, on new data
            filler.fill(arena, t)
            mon.step(arena, stats=stats)
            want = stats["norm"].cpu().numpy()
            out = torch.full((w.num_units,), float("nan"), dtype=torch.float64, device=cuda_device)
            st = _static_norms(lib, arena, w, out)
            assert st == N.GNMR_OK, N.last_error(None)
            torch.cuda.synchronize()
            got = out.cpu().numpy()
            np.testing.assert_allclose(got, want, rtol=RTOL, atol=0)
            # and against the oracle on the same bytes (Eq. local_gradient, summed in fp64)
            host.copy_(arena)
            view = host.view(torch.int16).numpy().view(np.uint16) if w.dtype == "bf16" else host.numpy()
            exact = oracle.unit_norms_threaded(view, w.offsets, w.lengths, 16)
            np.testing.assert_allclose(got, exact, rtol=RTOL, atol=0)
    finally:
        mon.close()


def test_static_norms_limits_and_errors(cuda_device):
    import torch
    lib = N.load()
    out = torch.empty(4, dtype=torch.float64, device=cuda_device)
    arena = torch.zeros(1 << 20, dtype=torch.float32, device=cuda_device)
    too_many = 131073
    off = np.zeros(too_many, np.int64)
    ln = np.ones(too_many, np.int64)
    st = lib.gnmr_unit_norms_static(arena.data_ptr(), arena.numel(), N.GNMR_DTYPE_F32, too_many,
                                    off.ctypes.data, ln.ctypes.data, out.data_ptr(), None)
    assert st == N.GNMR_ERR_INVALID_ARG and N.last_error(None) == "units > 131072"
    off = np.array([0, 5], np.int64)
    ln = np.array([5, 1 << 20], np.int64)
    st = lib.gnmr_unit_norms_static(arena.data_ptr(), arena.numel(), N.GNMR_DTYPE_F32, 2,
                                    off.ctypes.data, ln.ctypes.data, out.data_ptr(), None)
    assert st == N.GNMR_ERR_LAYOUT and N.last_error(None) == "unit off arena"
    # a valid call after the rejected ones still works
    ln = np.array([5, 7], np.int64)
    arena[:12] = 2.0
    st = lib.gnmr_unit_norms_static(arena.data_ptr(), arena.numel(), N.GNMR_DTYPE_F32, 2,
                                    off.ctypes.data, ln.ctypes.data, out.data_ptr(), None)
    assert st == N.GNMR_OK
    torch.cuda.synchronize()
    np.testing.assert_allclose(out[:2].cpu().numpy(), [np.sqrt(20.0), np.sqrt(28.0)], rtol=RTOL)


def test_static_norms_follow_layout_changes(cuda_device):
    """Calls alternate between two layouts (and one layout array is rewritten
    in place): each call's norms are those of its own layout, so the reuse of
    a previous call's uploaded tables never leaks into the next."""
    import torch
    import oracle
    lib = N.load()
    rng = np.random.default_rng(21)
    n = 1 << 20
    host = rng.standard_normal(n).astype(np.float32)
    arena = torch.from_numpy(host).to(cuda_device)
    layouts = []
    for U in (100, 37):
        ln = rng.integers(0, 40_000, U).astype(np.int64)
        off = rng.integers(0, n - 40_000, U).astype(np.int64)
        layouts.append((off, ln))
    out = torch.empty(100, dtype=torch.float64, device=cuda_device)
    for k in (0, 1, 0, 1, 0):
        off, ln = layouts[k]
        st = lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, len(off), off.ctypes.data,
                                        ln.ctypes.data, out.data_ptr(), None)
        assert st == N.GNMR_OK, N.last_error(None)
        torch.cuda.synchronize()
        want = oracle.unit_norms(host, off, ln)
        np.testing.assert_allclose(out[:len(off)].cpu().numpy(), want, rtol=RTOL, atol=0)
    off, ln = layouts[0]
    ln[::3] = 7                                      # same array objects, new contents
    st = lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, len(off), off.ctypes.data,
                                    ln.ctypes.data, out.data_ptr(), None)
    assert st == N.GNMR_OK
    torch.cuda.synchronize()
    np.testing.assert_allclose(out[:len(off)].cpu().numpy(), oracle.unit_norms(host, off, ln), rtol=RTOL, atol=0)


def test_static_norms_reject_tables_of_another_layout(cuda_device):
    """Calls that overlap on the GPU race on the shared array.  Here one call
    repeats the uploaded layout (so it enqueues no upload) behind a long
    sleep on one stream while a call with a different layout uploads and runs
    on another stream: when the first kernel finally runs, the tables belong
    to the other layout, and it writes NaN for every unit instead of reading
    them.  The second call's norms are correct."""
    import torch
    import oracle
    lib = N.load()
    rng = np.random.default_rng(23)
    n = 1 << 20
    host = rng.standard_normal(n).astype(np.float32)
    arena = torch.from_numpy(host).to(cuda_device)
    layouts = []
    for U in (80, 45):
        ln = rng.integers(1, 30_000, U).astype(np.int64)
        off = rng.integers(0, n - 30_000, U).astype(np.int64)
        layouts.append((off, ln))
    (off1, ln1), (off2, ln2) = layouts
    out1 = torch.zeros(80, dtype=torch.float64, device=cuda_device)
    out2 = torch.zeros(45, dtype=torch.float64, device=cuda_device)
    s1, s2 = torch.cuda.Stream(cuda_device), torch.cuda.Stream(cuda_device)
    assert lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, 80, off1.ctypes.data,
                                      ln1.ctypes.data, out1.data_ptr(), s1.cuda_stream) == N.GNMR_OK
    torch.cuda.synchronize()
    np.testing.assert_allclose(out1.cpu().numpy(), oracle.unit_norms(host, off1, ln1), rtol=RTOL, atol=0)
    with torch.cuda.stream(s1):
        torch.cuda._sleep(200_000_000)               # about 0.1 s on this GPU's clock
    assert lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, 80, off1.ctypes.data,
                                      ln1.ctypes.data, out1.data_ptr(), s1.cuda_stream) == N.GNMR_OK
    assert lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, 45, off2.ctypes.data,
                                      ln2.ctypes.data, out2.data_ptr(), s2.cuda_stream) == N.GNMR_OK
    s2.synchronize()
    s1.synchronize()
    np.testing.assert_allclose(out2.cpu().numpy(), oracle.unit_norms(host, off2, ln2), rtol=RTOL, atol=0)
    assert np.isnan(out1.cpu().numpy()).all()

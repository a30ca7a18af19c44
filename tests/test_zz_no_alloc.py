"""gnmr_unit_norms_static: per-unit norms for callers that cannot allocate
device memory (a framework's caching allocator owns the GPU, a hook runs in
the middle of a step where cudaMalloc's device synchronisation would stall
it, or the deployment fixes its footprint up front).  Its scratch is a static
device array inside libgnmr, so it needs no handle.

Called through the C ABI and checked against gnmr_step's own norm output
(stats->norm) on the same arena, twice in a row, within the tolerance of the
other parity tests.  Kept in its own file, collected last."""
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
    w = workloads.make(config, shrink=shrink, steps=3)
    filler = workloads.Filler(w, cuda_device)
    arena = filler.new_arena()
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


def test_static_norms_repeat_layout_is_graph_capturable(cuda_device):
    """Once a layout is on the device, a call repeating it enqueues no host
    copies: it is captured in a CUDA graph, and replays compute the norms of
    whatever the arena holds at replay time."""
    import torch
    import oracle
    lib = N.load()
    rng = np.random.default_rng(22)
    n = 1 << 20
    arena = torch.empty(n, dtype=torch.float32, device=cuda_device)
    off = np.sort(rng.integers(0, n - 50_000, 64)).astype(np.int64)
    ln = rng.integers(1, 50_000, 64).astype(np.int64)
    out = torch.empty(64, dtype=torch.float64, device=cuda_device)
    stream = torch.cuda.Stream(cuda_device)

    def call():
        return lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_F32, 64, off.ctypes.data,
                                          ln.ctypes.data, out.data_ptr(), stream.cuda_stream)

    arena.normal_()
    assert call() == N.GNMR_OK                       # uploads the layout
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        assert call() == N.GNMR_OK
    for scale in (0.5, 3.0):
        host = (rng.standard_normal(n) * scale).astype(np.float32)
        arena.copy_(torch.from_numpy(host))
        torch.cuda.synchronize()
        graph.replay()
        torch.cuda.synchronize()
        np.testing.assert_allclose(out.cpu().numpy(), oracle.unit_norms(host, off, ln), rtol=RTOL, atol=0)

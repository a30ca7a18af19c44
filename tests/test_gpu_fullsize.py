"""Parity at the workloads' full sizes and step counts, in the launch
configuration bench.py times (same Monitor construction, same device plan).
The oracle computes every unit's norm from the full arena each step (copied
to the host), so every output is compared, not a sample."""
import pytest

import workloads
from paper_2606_00539_gb300 import Monitor
from tests import trace_driver as TD

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _bench_monitor(w):
    # exactly as bench.py builds it
    return Monitor(w.offsets, w.lengths, device=0, **w.monitor_kwargs())


@pytest.mark.parametrize("config", ["llama2-1.3b", "llama2-13b", "moe", "aq-stress"])
def test_full_size_parity(config, cuda_device):
    w = workloads.make(config)
    tr = TD.LockstepTrace(w, "cuda:0", _bench_monitor)
    try:
        info = tr.mon.info()
        assert info["num_units"] == w.num_units
        selected = 0
        for t in range(w.steps):
            norms, res, got = tr.step(t)
            TD.compare(norms, res, got, 1e-5)
            selected += res.n_selected
        assert selected > 0, "the trace should exercise the recovery path"
    finally:
        tr.close()


def test_unit_longer_than_2_pow_31_elements(cuda_device):
    """One bf16 unit of 2^31 + 777 elements (4.3 GB, a single huge tensor)
    between small units at odd offsets: 64-bit element indexing in the plan,
    the warp runs and the allocation-free path; norms against the oracle."""
    import numpy as np
    import torch

    import oracle
    from paper_2606_00539_gb300 import _native as N
    big = (1 << 31) + 777
    n = big + 5 + 4099
    arena = torch.empty(n, dtype=torch.bfloat16, device=cuda_device)
    gen = torch.Generator(device=cuda_device).manual_seed(7)
    for s0 in range(0, n, 1 << 28):
        k = min(1 << 28, n - s0)
        arena[s0:s0 + k] = torch.randn(k, generator=gen, device=cuda_device).to(torch.bfloat16)
    off = np.array([0, 5, 5 + big, 5 + big + 3], np.int64)
    ln = np.array([5, big, 3, 4096], np.int64)
    host = arena.cpu().view(torch.int16).numpy().view(np.uint16)
    want = oracle.unit_norms_threaded(host, off, ln, 16)
    mon = Monitor(off, ln, dtype="bf16", device=0)
    stats = mon.new_stats()
    try:
        mon.step(arena, stats=stats)
        got = stats["norm"].cpu().numpy()
    finally:
        mon.close()
    np.testing.assert_allclose(got, want, rtol=1e-5, atol=0)
    out = torch.empty(4, dtype=torch.float64, device=cuda_device)
    lib = N.load()
    assert lib.gnmr_unit_norms_static(arena.data_ptr(), n, N.GNMR_DTYPE_BF16, 4, off.ctypes.data,
                                      ln.ctypes.data, out.data_ptr(), None) == N.GNMR_OK
    torch.cuda.synchronize()
    np.testing.assert_allclose(out.cpu().numpy(), want, rtol=1e-5, atol=0)

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

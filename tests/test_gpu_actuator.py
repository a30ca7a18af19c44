"""The recovery actuator on the GPU against the oracle's fake quantization
(App. E.2): every output bit must match, for both dtypes, every format,
mixed per-unit formats chosen by a mask, unaligned rows, special rows, in
place, and with the mask written by gnmr_step."""
import numpy as np
import pytest

import oracle
import workloads
from paper_2606_00539_gb300 import Monitor
from paper_2606_00539_gb300 import _native as N

pytestmark = pytest.mark.gpu

FORMATS = [N.GNMR_FQ_E2M1, N.GNMR_FQ_E3M2, N.GNMR_FQ_E4M3, N.GNMR_FQ_E5M2, N.GNMR_FQ_NONE]


def _layout(rng, U, max_rows=40, max_cols=700, gap=True):
    rows = rng.integers(0, max_rows, U).astype(np.int64)
    cols = rng.integers(1, max_cols, U).astype(np.int64)
    off, pos = [], 0
    for r, c in zip(rows, cols):
        pos += int(rng.integers(0, 5)) if gap else 0          # odd starts on purpose
        off.append(pos)
        pos += int(r * c)
    return np.array(off, np.int64), rows, cols, pos + 3


def _host_bits(t):
    import torch
    t = t.cpu()
    return t.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else t.numpy()


def _oracle_apply(host_in, off, rows, cols, fmt_of_unit):
    out = host_in.copy()
    for b in range(len(off)):
        n = int(rows[b] * cols[b])
        if n == 0:
            continue
        blk = host_in[off[b]:off[b] + n].reshape(rows[b], cols[b])
        out[off[b]:off[b] + n] = oracle.fake_quant(blk, fmt_of_unit[b]).reshape(-1)
    return out


def _special_rows(x, off, rows, cols):
    """Plant zero, NaN, Inf, -0, huge-range and tiny rows in the first units
    (the tiny row's amax, 1e-37, makes fmax / amax overflow fp32 for E4M3
    and E5M2: that row must come back unchanged, with no NaN)."""
    import torch
    for b, kind in enumerate(["zero", "nan", "inf", "negzero", "wide", "tiny"]):
        if b >= len(off) or rows[b] == 0:
            continue
        s, c = int(off[b]), int(cols[b])
        if kind == "zero":
            x[s:s + c] = 0
        elif kind == "nan":
            x[s + c // 2] = float("nan")
        elif kind == "inf":
            x[s] = float("-inf")
        elif kind == "negzero":
            x[s:s + c] = -0.0
        elif kind == "wide":
            x[s:s + c] = torch.logspace(-30, 30, c, dtype=torch.float32).to(x.dtype) * \
                torch.sign(torch.randn(c)).to(x.dtype)
        else:
            row = torch.randn(c, dtype=torch.float32) * 1e-37
            row[::4] = 0.0
            row[0] = 1e-37
            x[s:s + c] = row.to(x.dtype)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("low,rec", [(N.GNMR_FQ_E2M1, N.GNMR_FQ_E4M3), (N.GNMR_FQ_E3M2, N.GNMR_FQ_E5M2),
                                     (N.GNMR_FQ_E4M3, N.GNMR_FQ_NONE)])
def test_actuator_bit_exact(dtype, low, rec, cuda_device):
    import torch
    rng = np.random.default_rng(low * 10 + rec)
    U = 60
    off, rows, cols, total = _layout(rng, U)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    x = (torch.randn(total, generator=torch.Generator().manual_seed(3)) *
         torch.exp(torch.randn(total, generator=torch.Generator().manual_seed(4)))).to(tdt)
    _special_rows(x, off, rows, cols)
    d_in = x.to(cuda_device)
    d_out = torch.full_like(d_in, 7.0)
    mask = (rng.random(U) < 0.4).astype(np.uint8)
    d_mask = torch.from_numpy(mask).to(cuda_device)
    h = N.gnmr_actuator_create(off, rows, cols, N.GNMR_DTYPE_BF16 if dtype == "bf16" else N.GNMR_DTYPE_F32, 0)
    try:
        N.gnmr_actuator_apply(h, d_in.data_ptr(), d_out.data_ptr(), total, d_mask.data_ptr(), low, rec)
        torch.cuda.synchronize()
        got = _host_bits(d_out)
        want = _oracle_apply(_host_bits(x), off, rows, cols, [rec if m else low for m in mask])
        covered = np.zeros(total, bool)
        for b in range(U):
            covered[off[b]:off[b] + rows[b] * cols[b]] = True
        g, w_ = got[covered], want[covered]
        same = (g.view(np.uint16 if dtype == "bf16" else np.uint32) ==
                w_.view(np.uint16 if dtype == "bf16" else np.uint32))
        assert same.all(), f"{(~same).sum()} of {same.size} elements differ"
        # bytes outside every unit are untouched
        seven = _host_bits(torch.full((1,), 7.0, dtype=tdt))[0]
        assert np.all(_host_bits(d_out)[~covered] == seven)
        # in place, mask NULL = low-cost everywhere
        N.gnmr_actuator_apply(h, d_in.data_ptr(), d_in.data_ptr(), total, None, low, rec)
        torch.cuda.synchronize()
        want2 = _oracle_apply(_host_bits(x), off, rows, cols, [low] * U)
        g2 = _host_bits(d_in)[covered]
        w2 = want2[covered]
        assert np.array_equal(g2.view(np.uint16 if dtype == "bf16" else np.uint32),
                              w2.view(np.uint16 if dtype == "bf16" else np.uint32))
    finally:
        N.gnmr_actuator_destroy(h)


def test_actuator_driven_by_gnmr_step(cuda_device):
    """The mask gnmr_step writes selects each unit's activation format."""
    import torch
    w = workloads.make("llama2-13b", shrink=64, steps=8)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    mon = Monitor(w.offsets, w.lengths, device=0, **w.monitor_kwargs())
    rng = np.random.default_rng(1)
    rows = np.full(w.num_units, 32, np.int64)
    cols = (w.lengths // 64).clip(1)
    off = np.concatenate([[0], np.cumsum(rows * cols)[:-1]]).astype(np.int64)
    total = int((rows * cols).sum())
    acts = torch.randn(total, device=cuda_device).to(torch.bfloat16)
    out = torch.empty_like(acts)
    h = N.gnmr_actuator_create(off, rows, cols, N.GNMR_DTYPE_BF16, 0)
    try:
        for t in range(w.steps):
            f.fill(arena, t)
            mask = mon.step(arena)
            N.gnmr_actuator_apply(h, acts.data_ptr(), out.data_ptr(), total, mask.data_ptr(),
                                  N.GNMR_FQ_E2M1, N.GNMR_FQ_E4M3,
                                  torch.cuda.current_stream().cuda_stream)
            torch.cuda.synchronize()
            m = mask.cpu().numpy()
            want = _oracle_apply(_host_bits(acts), off, rows, cols,
                                 [N.GNMR_FQ_E4M3 if v else N.GNMR_FQ_E2M1 for v in m])
            assert np.array_equal(_host_bits(out), want)
        del rng
    finally:
        N.gnmr_actuator_destroy(h)
        mon.close()


def test_actuator_errors(cuda_device):
    import torch
    off = np.array([0, 10], np.int64)
    rows = np.array([2, 3], np.int64)
    cols = np.array([5, 4], np.int64)
    with pytest.raises(N.GnmrError):
        N.gnmr_actuator_create(np.array([-1, 0]), rows, cols, N.GNMR_DTYPE_F32, 0)
    h = N.gnmr_actuator_create(off, rows, cols, N.GNMR_DTYPE_F32, 0)
    x = torch.zeros(22, device=cuda_device)
    try:
        with pytest.raises(N.GnmrError) as ei:
            N.gnmr_actuator_apply(h, x.data_ptr(), x.data_ptr(), 21, None, 1, 3)
        assert ei.value.status == N.GNMR_ERR_LAYOUT
        with pytest.raises(N.GnmrError) as ei:
            N.gnmr_actuator_apply(h, x.data_ptr(), x.data_ptr(), 22, None, 9, 3)
        assert ei.value.status == N.GNMR_ERR_INVALID_ARG
        N.gnmr_actuator_apply(h, x.data_ptr(), x.data_ptr(), 22, None, 1, 3)
    finally:
        N.gnmr_actuator_destroy(h)

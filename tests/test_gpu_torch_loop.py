"""The monitor and the actuator inside a real PyTorch training loop.

A small MLP's parameter gradients (fp32, or bf16 for a bf16 model) live in
one flat arena (every
`.grad` is a view of it, so backward writes straight into the arena); each
Linear's weight and bias form one block-level unit.  Every step: the
monitor's norms against torch's own norms of the same gradients, its
decisions against the oracle stepped on those norms (where no decision is
within rounding of a threshold), and the actuator, driven by the mask, on
the layers' saved inputs against the oracle's fake quantization."""
import numpy as np
import pytest

import oracle
from paper_2606_00539_gb300 import Monitor
from paper_2606_00539_gb300 import _native as N

pytestmark = pytest.mark.gpu

KW = dict(window=3, max_o=2, lock_len=2, warmup_steps=2)
ALPHA, BETA = (1.5, 1.2), (1.5, 1.5)


def _has_margin(res, max_o, rel=1e-4):
    r = res.risk[np.isfinite(res.risk)]
    if np.any(np.abs(r - 1.0) < rel * np.maximum(1.0, r)):
        return False
    cand = np.sort(res.risk[res.risk > 1.0])[::-1]
    if len(cand) > max_o > 0:
        a, b = cand[max_o - 1], cand[max_o]
        return (a - b) > rel * a
    return True


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_training_loop_with_monitor_and_actuator(dtype, cuda_device):
    import torch
    torch.manual_seed(0)
    dev = cuda_device
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    ebytes = 2 if dtype == "bf16" else 4
    align = 16 // ebytes
    layers = [torch.nn.Linear(64, 96), torch.nn.Linear(96, 96), torch.nn.Linear(96, 96), torch.nn.Linear(96, 10)]
    model = torch.nn.Sequential(layers[0], torch.nn.ReLU(), layers[1], torch.nn.ReLU(),
                                layers[2], torch.nn.ReLU(), layers[3]).to(dev, tdt)
    params = list(model.parameters())                 # w0, b0, w1, b1, ...
    offs, lens, seg_unit, pos = [], [], [], 0
    for i, p in enumerate(params):
        offs.append(pos)
        lens.append(p.numel())
        seg_unit.append(i // 2)                       # a layer's weight and bias: one unit
        pos += (p.numel() + align - 1) // align * align   # 16-byte aligned starts
    arena = torch.zeros(pos, dtype=tdt, device=dev)
    for p, o in zip(params, offs):
        p.grad = arena[o:o + p.numel()].view_as(p)
    U = len(layers)
    mon = Monitor(np.array(offs, np.int64), np.array(lens, np.int64), dtype=dtype, device=0,
                  segment_unit=np.array(seg_unit, np.int32), num_units=U, alpha=ALPHA, beta=BETA, **KW)
    ctl = oracle.Controller(U, alpha=ALPHA, beta=BETA, **KW)
    stats = mon.new_stats()

    acts = {}
    hooks = [l.register_forward_hook(lambda m, inp, out, i=i: acts.__setitem__(i, inp[0].detach()))
             for i, l in enumerate(layers)]
    rows = 256
    cols = np.array([l.in_features for l in layers], np.int64)
    a_off = np.concatenate([[0], np.cumsum(rows * cols)[:-1]]).astype(np.int64)
    act = N.gnmr_actuator_create(a_off, np.full(U, rows, np.int64), cols,
                                 N.GNMR_DTYPE_BF16 if dtype == "bf16" else N.GNMR_DTYPE_F32, 0)
    opt = torch.optim.SGD(model.parameters(), lr=0.05)
    gen = torch.Generator().manual_seed(1)
    X = torch.randn(rows, 64, generator=gen).to(dev, tdt)
    Y = torch.randint(0, 10, (rows,), generator=gen).to(dev)
    compared = selected = 0
    try:
        for step in range(12):
            xb = X * (40.0 if step in (6, 7) else 1.0)       # a burst of large gradients
            arena.zero_()
            loss = torch.nn.functional.cross_entropy(model(xb), Y)
            loss.backward()
            assert all(p.grad.data_ptr() == arena.data_ptr() + ebytes * o for p, o in zip(params, offs))
            mask = mon.step(arena, stats=stats)
            want_n = np.array([np.sqrt(sum(float(params[j].grad.double().pow(2).sum()) for j in (2 * u, 2 * u + 1)))
                               for u in range(U)])
            np.testing.assert_allclose(stats["norm"].cpu().numpy(), want_n, rtol=1e-5, atol=0)
            res = ctl.step(want_n)
            np.testing.assert_allclose(stats["risk"].cpu().numpy(), res.risk, rtol=1e-5, atol=0)
            got_mask = mask.cpu().numpy()
            if _has_margin(res, KW["max_o"]):
                compared += 1
                assert np.array_equal(got_mask, res.mask), f"step {step + 1}: mask"
                assert np.array_equal(stats["lock"].cpu().numpy(), res.lock), f"step {step + 1}: lock"
            selected += int(got_mask.sum())
            # the actuator on the layers' saved inputs: recovery format (E4M3) where the mask is set
            a_in = torch.cat([acts[i].reshape(-1) for i in range(U)]).contiguous()
            a_out = torch.empty_like(a_in)
            N.gnmr_actuator_apply(act, a_in.data_ptr(), a_out.data_ptr(), a_in.numel(), mask.data_ptr(),
                                  N.GNMR_FQ_E2M1, N.GNMR_FQ_E4M3)
            bits = (lambda t: t.cpu().view(torch.int16).numpy().view(np.uint16)) if dtype == "bf16" \
                else (lambda t: t.cpu().numpy())
            host_in, host_out = bits(a_in), bits(a_out)
            for u in range(U):
                blk = slice(int(a_off[u]), int(a_off[u] + rows * cols[u]))
                code = N.GNMR_FQ_E4M3 if got_mask[u] else N.GNMR_FQ_E2M1
                want = oracle.fake_quant(host_in[blk].reshape(rows, int(cols[u])), code)
                assert np.array_equal(host_out[blk].view(np.uint8), want.reshape(-1).view(np.uint8)), \
                    f"step {step + 1}, unit {u}: actuator"
            opt.step()
    finally:
        for h in hooks:
            h.remove()
        N.gnmr_actuator_destroy(act)
        mon.close()
        ctl.close()
    assert compared >= 6
    assert selected > 0                              # the burst put units on the recovery path

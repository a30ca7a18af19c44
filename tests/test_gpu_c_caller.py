"""The C ABI from a plain C11 program (tests/c_caller.c): no Python and no
torch in the process that calls libgnmr.  The program is compiled with gcc
against include/gnmr.h, linked with libgnmr.so and the CUDA runtime, fed a
seeded multi-step fp32 trace through a file, and its masks, locks, counts
and statistics are compared with the oracle step by step."""
import glob
import os
import subprocess
from types import SimpleNamespace

import numpy as np
import pytest

import oracle
from paper_2606_00539_gb300 import build as B
from tests import trace_driver as TD

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2606_00539_gb300")
RTOL = 1e-5


def _cuda_lib_dir(home):
    for cand in [os.path.join(home, "lib64")] + sorted(glob.glob(os.path.join(home, "targets", "*", "lib"))):
        if glob.glob(os.path.join(cand, "libcudart.so*")):
            return cand
    pytest.skip("libcudart.so not found")


def _compile(tmp_path):
    home = B._cuda_home()
    lib = _cuda_lib_dir(home)
    exe = str(tmp_path / "c_caller")
    subprocess.check_call(["gcc", "-std=c11", "-O1", "-Wall", "-I", os.path.join(ROOT, "include"),
                           "-I", os.path.join(home, "include"), os.path.join(ROOT, "tests", "c_caller.c"),
                           "-o", exe, "-L", PKG, "-lgnmr", "-L", lib, "-lcudart",
                           "-Wl,-rpath," + PKG, "-Wl,-rpath," + lib])
    return exe


def _trace(rng, U, steps, cfg):
    """Packed fp32 units with gaps, per-(step, unit) levels and a few spikes,
    each step's levels redrawn where the oracle's decisions lack margin.
    Returns offsets, lengths, arenas [steps][n] and the oracle's results."""
    lengths = rng.integers(0, 9000, U).astype(np.int64)
    lengths[::37] = 0
    gaps = rng.integers(0, 5, U)
    offsets = np.zeros(U, np.int64)
    pos = 0
    for b in range(U):
        pos += int(gaps[b])
        offsets[b] = pos
        pos += int(lengths[b])
    n = pos + 3
    base = rng.standard_normal(n).astype(np.float32)
    unit_of = np.full(n, -1, np.int64)
    for b in range(U):
        unit_of[offsets[b]:offsets[b] + lengths[b]] = b
    levels = np.exp(0.35 * rng.standard_normal((steps, U)))
    for _ in range(12):
        levels[rng.integers(3, steps), rng.integers(0, U)] *= float(rng.uniform(5, 40))
    ctl = oracle.Controller(U, window=cfg.window, max_o=cfg.max_o, lock_len=cfg.lock_len,
                            alpha=cfg.alpha, beta=cfg.beta, eps=cfg.eps)
    margin = SimpleNamespace(recoverable=np.ones(U, np.uint8), warmup_steps=0, alpha=cfg.alpha,
                             beta=cfg.beta, window=cfg.window, max_o=cfg.max_o)
    arenas, expect = [], []
    try:
        for t in range(steps):
            for attempt in range(40):
                scale = np.ones(n, np.float32)
                inside = unit_of >= 0
                scale[inside] = levels[t, unit_of[inside]].astype(np.float32)
                x = base * scale
                norms = oracle.unit_norms(x, offsets, lengths)
                before = ctl.get_state()
                res = ctl.step(norms)
                bad = TD.margin_violations(before, res, margin, t + 1)
                if not bad:
                    break
                ctl.set_state(before)
                levels[t, bad] *= np.exp(0.05 * rng.standard_normal(len(bad)))
            else:
                raise AssertionError(f"no decision margin at step {t + 1}")
            arenas.append(x)
            expect.append((norms, res))
    finally:
        ctl.close()
    return offsets, lengths, np.stack(arenas), expect


def _parse(text, U):
    lines = text.splitlines()
    steps = []
    i = 0
    while i < len(lines):
        head = lines[i].split()
        assert head[0] == "step" and head[2] == "counts", lines[i]
        rows = [ln.split() for ln in lines[i + 1:i + 1 + U]]
        got = {"counts": [int(head[3]), int(head[4])],
               "mask": np.array([int(r[1]) for r in rows], np.uint8),
               "lock": np.array([int(r[2]) for r in rows], np.int32)}
        for k, name in enumerate(("norm", "gnmr", "dgnmr", "risk")):
            got[name] = np.array([float.fromhex(r[3 + k]) for r in rows])
        steps.append(got)
        i += 1 + U
    return steps


def test_c_program_matches_the_oracle(tmp_path, cuda_device):
    exe = _compile(tmp_path)
    rng = np.random.default_rng(41)
    U, steps = 257, 24
    cfg = SimpleNamespace(window=4, max_o=6, lock_len=3, alpha=(1.3, 1.3), beta=(1.4, 1.4), eps=1e-8)
    offsets, lengths, arenas, expect = _trace(rng, U, steps, cfg)
    path = tmp_path / "trace.bin"
    with open(path, "wb") as f:
        f.write(np.array([U, arenas.shape[1], steps, cfg.window, cfg.max_o, cfg.lock_len], "<i8").tobytes())
        f.write(np.array([cfg.alpha[0], cfg.beta[0], cfg.eps], "<f8").tobytes())
        f.write(offsets.astype("<i8").tobytes())
        f.write(lengths.astype("<i8").tobytes())
        f.write(arenas.astype("<f4").tobytes())
    out = subprocess.run([exe, str(path)], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    got = _parse(out.stdout, U)
    assert len(got) == steps
    selected = 0
    for (norms, res), g in zip(expect, got):
        TD.compare(norms, res, g, RTOL)
        selected += res.n_selected
    assert selected > 0, "the trace should exercise the recovery path"

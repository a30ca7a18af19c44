"""Pins for the oracle's fake quantization (the recovery actuator, App. E.2):
rounding is checked against a brute-force search over every encoding of each
format, enumerated from the minifloat definitions (sign, exponent with bias,
mantissa; subnormals at exponent code 0), with ties to the even code; the
per-token scaling against its closed-form consequences."""
import math

import numpy as np
import pytest

import oracle

# (code, exponent bits, mantissa bits, bias, exclude top exponent code, max)
FORMATS = {
    oracle.FQ_E2M1: (2, 1, 1, False, 6.0),
    oracle.FQ_E3M2: (3, 2, 3, False, 28.0),
    oracle.FQ_E4M3: (4, 3, 7, "nan_only", 448.0),
    oracle.FQ_E5M2: (5, 2, 15, True, 57344.0),
}


def _encodings(code):
    """All non-negative finite values of the format with their mantissa code."""
    eb, mb, bias, top, _ = FORMATS[code]
    vals = []
    for E in range(1 << eb):
        for m in range(1 << mb):
            if top is True and E == (1 << eb) - 1:
                continue                                   # E5M2: inf / NaN
            if top == "nan_only" and E == (1 << eb) - 1 and m == (1 << mb) - 1:
                continue                                   # E4M3: the single NaN code
            if E == 0:
                v = math.ldexp(m / (1 << mb), 1 - bias)
            else:
                v = math.ldexp(1 + m / (1 << mb), E - bias)
            vals.append((v, (E << mb) | m))
    return sorted(vals)


@pytest.mark.parametrize("code", sorted(FORMATS))
def test_format_max_and_grid(code):
    vals = _encodings(code)
    assert vals[-1][0] == FORMATS[code][4]
    for v, _ in vals:                         # every representable value is a fixed point
        assert oracle.fq_round(v, code) == v
        assert oracle.fq_round(-v, code) == -v


@pytest.mark.parametrize("code", sorted(FORMATS))
def test_rounding_is_nearest_with_ties_to_even(code):
    vals = _encodings(code)
    grid = np.array([v for v, _ in vals])
    codes = {v: c for v, c in vals}
    rng = np.random.default_rng(code)
    fmax = FORMATS[code][4]
    # random values over the whole range, plus every midpoint (the ties)
    xs = list(np.float32(rng.uniform(0, fmax * 1.2, 4000)))
    xs += list(np.float32(np.exp(rng.uniform(math.log(grid[1] / 4), math.log(fmax), 4000))))
    xs += [np.float32((a + b) / 2) for a, b in zip(grid[:-1], grid[1:])]
    for x in xs:
        x = float(x)
        if x >= fmax:
            want = fmax
        else:
            d = np.abs(grid - x)
            best = np.nonzero(d == d.min())[0]
            if len(best) == 1:
                want = grid[best[0]]
            else:                              # tie: the even code
                want = [grid[i] for i in best if codes[grid[i]] % 2 == 0][0]
        assert oracle.fq_round(x, code) == want, (code, x)
        assert oracle.fq_round(-x, code) == -want


def test_per_token_scaling_closed_forms():
    rng = np.random.default_rng(9)
    x = (rng.standard_normal((64, 96)) * np.exp(rng.standard_normal((64, 1)))).astype(np.float32)
    x[3] = 0.0
    for code in sorted(FORMATS):
        y = oracle.fake_quant(x, code)
        fmax = np.float32(FORMATS[code][4])
        assert np.all(y[3] == 0.0)                                 # zero token stays zero
        amax = np.max(np.abs(x), axis=1)
        ymax = np.max(np.abs(y), axis=1)
        nz = amax > 0
        # the largest element maps to fmax and back: within one rounding of itself
        np.testing.assert_allclose(ymax[nz], amax[nz], rtol=1e-6)
        # every output is a grid value times the token's scale
        scale = (amax / fmax).astype(np.float32)
        grid = np.array([v for v, _ in _encodings(code)], np.float32)
        for r in np.nonzero(nz)[0][:8]:
            q = np.abs(y[r]) / scale[r]
            assert np.all(np.min(np.abs(q[:, None] - grid[None, :]), axis=1) <= 1e-5 * fmax)
    # format 0 copies; a token with a non-finite value passes through
    assert np.array_equal(oracle.fake_quant(x, oracle.FQ_NONE), x)
    z = x.copy()
    z[5, 7] = np.inf
    z[6, 0] = np.nan
    yz = oracle.fake_quant(z, oracle.FQ_E2M1)
    assert np.array_equal(yz[5], z[5]) and np.array_equal(yz[6], z[6], equal_nan=True)
    assert np.array_equal(yz[7], oracle.fake_quant(x, oracle.FQ_E2M1)[7])


@pytest.mark.parametrize("code", sorted(FORMATS))
def test_rows_whose_scale_factor_overflows_are_kept(code):
    """A row with a finite amax below fmax / FLT_MAX would get the scale
    factor inv = fmax / amax = +inf in fp32, turning its zeros into NaN
    (0 * inf).  Such a row is kept bit for bit, like a zero row; a row just
    above that bound is quantized as usual (finite, its max maps back to
    within one rounding of itself)."""
    torch = pytest.importorskip("torch")
    fmax = np.float32(FORMATS[code][4])
    bound = fmax / np.finfo(np.float32).max             # inv overflows below this amax
    rng = np.random.default_rng(11)
    with np.errstate(over="ignore"):
        _overflow_rows(code, fmax, bound, rng, torch)


def _overflow_rows(code, fmax, bound, rng, torch):
    for amax, kept in ((np.float32(bound * 0.5), True), (np.float32(bound * 4.0), False),
                       (np.float32(1e-37), bool(np.isinf(np.float32(fmax) / np.float32(1e-37))))):
        x = (rng.uniform(-1.0, 1.0, (3, 50)) * amax).astype(np.float32)
        x[:, ::5] = 0.0                                  # zeros that 0 * inf would make NaN
        x[:, 1] = amax
        y = oracle.fake_quant(x, code)
        assert not np.isnan(y).any()
        if kept:
            assert np.array_equal(y.view(np.uint32), x.view(np.uint32))
        else:
            assert np.all(np.isfinite(y)) and np.all(y[:, ::5] == 0.0)
            np.testing.assert_allclose(np.max(np.abs(y), axis=1), amax, rtol=1e-6)
        # the same rows as bf16 bit patterns
        xb = torch.from_numpy(x).to(torch.bfloat16)
        bits = xb.view(torch.int16).numpy().view(np.uint16)
        amax_b = float(xb.abs().max())
        yb = oracle.fake_quant(bits, code)
        yf = torch.from_numpy(yb.view(np.int16)).view(torch.bfloat16).float().numpy()
        assert not np.isnan(yf).any()
        if np.isinf(np.float32(fmax) / np.float32(amax_b)):
            assert np.array_equal(yb, bits)


def test_bf16_rows():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(10)
    xf = rng.standard_normal((16, 40)).astype(np.float32)
    xb = torch.from_numpy(xf).to(torch.bfloat16)
    bits = xb.view(torch.int16).numpy().view(np.uint16)
    yb = oracle.fake_quant(bits, oracle.FQ_E3M2)
    y_from_f32 = oracle.fake_quant(xb.float().numpy(), oracle.FQ_E3M2)
    want = torch.from_numpy(y_from_f32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(yb, want)       # bf16 path = fp32 path + RNE to bf16 (torch's rounding)

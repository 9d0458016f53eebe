"""Pins of the oracle's rounding to the weight storage dtype (no GPU)."""

import numpy as np
import torch

from oracle import rounding


def _torch_bf16(x64):
    # torch rounds fp32 -> bf16 with round-to-nearest-even; inputs here are
    # exactly representable in fp32, so no double rounding is involved.
    t = torch.from_numpy(np.asarray(x64, np.float32))
    return t.to(torch.bfloat16).to(torch.float64).numpy()


def test_bf16_matches_library_cast_on_fp32_inputs():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(200_000).astype(np.float32).astype(np.float64)
    x *= np.exp2(rng.integers(-140, 120, x.size))
    x = x.astype(np.float32).astype(np.float64)    # back into fp32 range / values
    x = x[np.isfinite(x)]
    assert np.array_equal(rounding.round_to_bf16(x), _torch_bf16(x))


def test_bf16_ties_go_to_even():
    one = 1.0
    ulp = 2.0 ** -7
    cases = {
        one + ulp / 2: one,                 # tie, 1.0 has even mantissa
        one + 3 * ulp / 2: one + 2 * ulp,   # tie, rounds up to even
        one + ulp / 2 + 2 ** -30: one + ulp,
        -(one + ulp / 2): -one,
        2.0 ** -126 * (1 + 2 ** -8): 2.0 ** -126,   # normal boundary tie
        2.0 ** -134: 0.0,                   # half the smallest subnormal -> even (0)
        3 * 2.0 ** -134: 2 * 2.0 ** -133,
    }
    for x, want in cases.items():
        assert rounding.round_to_bf16(np.array([x]))[0] == want, x


def test_bf16_overflow_and_specials():
    big = (2.0 - 2.0 ** -8) * 2.0 ** 127        # tie between max and 2^128 -> inf (even)
    out = rounding.round_to_bf16(np.array([big, -big, 0.0, -0.0, np.inf, np.nan]))
    assert out[0] == np.inf and out[1] == -np.inf
    assert out[2] == 0.0 and np.signbit(out[3]) and out[4] == np.inf and np.isnan(out[5])


def test_bf16_is_idempotent_and_within_half_ulp():
    rng = np.random.default_rng(1)
    x = rng.standard_normal(100_000) * 0.02
    y = rounding.round_to_bf16(x)
    assert np.array_equal(rounding.round_to_bf16(y), y)
    assert np.all(np.abs(y - x) <= rounding.bf16_ulp(y) / 2 * (1 + 1e-12))


def test_bf16_bit_helpers_roundtrip():
    rng = np.random.default_rng(2)
    y = rounding.round_to_bf16(rng.standard_normal(1000))
    assert np.array_equal(rounding.bf16_bits_to_f64(rounding.f64_to_bf16_bits(y)), y)


def test_f32_and_f64_modes():
    x = np.array([1.0 + 2.0 ** -30, 0.1])
    assert np.array_equal(rounding.round_to(x, "f32"), x.astype(np.float32).astype(np.float64))
    assert np.array_equal(rounding.round_to(x, "f64"), x)

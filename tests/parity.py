"""Comparison helpers for the parity tests (tolerances of the weight path)."""

import numpy as np

from oracle import rounding

# fp32 weights, moments: |d| <= REL * max(|x_oracle|, FLOOR * max|x_oracle|)
REL = 1e-5
FLOOR = 1e-3
# U, V: max abs difference
UV_ABS = 1e-5
# Box-Muller normals: fp32 log/sqrt/sincospi against fp64
NORMAL_ABS = 2e-6


def to_f64(t):
    import torch
    return t.detach().to("cpu", torch.float64).numpy() if t.dtype != torch.bfloat16 else \
        t.detach().to("cpu").to(torch.float32).to(torch.float64).numpy()


def rel_ok(got, want, rel=REL, floor=FLOOR):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    scale = np.maximum(np.abs(want), floor * (np.abs(want).max() if want.size else 0.0))
    bad = np.abs(got - want) > rel * scale
    return not bad.any(), int(bad.sum())


def assert_rel(got, want, what, rel=REL, floor=FLOOR):
    ok, nbad = rel_ok(got, want, rel, floor)
    if not ok:
        d = np.abs(np.asarray(got) - np.asarray(want))
        raise AssertionError(f"{what}: {nbad} elements beyond rel {rel} (max abs diff {d.max():.3e})")


def assert_weights(got, want, dtype, what):
    """bf16: |d| <= 1 ulp of the oracle's rounded value; fp32: relative 1e-5 (floored)."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    if dtype == "bf16":
        d = np.abs(got - want)
        ulp = rounding.bf16_ulp(want)
        bad = d > ulp
        if bad.any():
            raise AssertionError(f"{what}: {int(bad.sum())} bf16 elements more than 1 ulp off "
                                 f"(max {float((d / ulp).max()):.2f} ulp)")
        return int((d > 0).sum())
    assert_rel(got, want, what)
    return int((got != want).sum())

"""Comparison helpers for the parity tests (tolerances of the weight path).

Readings of the stated tolerances (bf16 weights within 1 ulp, fp32 weights and
Adam moments within relative 1e-5, U and V within 1e-5 absolute):

* a relative or ulp bound is taken at the magnitude of the OPERANDS of the
  operation that produced the value, not of the result alone.  When an update
  cancels most of a weight (W + delta ~ 0), or delta = sum_k U_ik P_kj cancels
  most of its own terms, the result's own ulp is arbitrarily small, while any
  fp32 evaluation carries an error proportional to the terms it summed; the
  operand scale is the one that bounds the arithmetic.
    weights: scale = max(|W_oracle|, |W_before|, T),  T = |U| |C| |V|^T
             plus TZ = eps sum|c_k| NORMAL_ABS (sum_a |U_ia|)(sum_b |V_jb|), the
             part of delta that the fp32 Gaussians may differ by
    moments: scale = beta |M_prev| + (1 - beta) Gabs   (Gabs = (1/q) sum_k |rho_k| |Z_k|)
             scale = beta2 |Vm_prev| + (1 - beta2) Gabs^2
* multi-step trajectories (state carried across many calls) are compared
  normwise: |d| <= 1e-5 * max |x_oracle| over the matrix.
"""

import numpy as np

from oracle import rng, rounding

REL = 1e-5
UV_ABS = 1e-5
# Box-Muller normals: fp32 log/sqrt/sincospi against fp64.  With |log error| <= 1 ulp,
# a correctly rounded sqrt and <= 1 ulp sin/cos, |dz| <= sqrt(-2 ln 2^-24) * (a few fp32
# ulps) ~ 5.77 * 4 * 6e-8 ~ 1.4e-6
NORMAL_ABS = 2e-6


def to_f64(t):
    import torch
    if t.dtype == torch.bfloat16:
        t = t.float()
    return t.detach().to("cpu", torch.float64).numpy()


def _report(d, tol, what):
    bad = d > tol
    if bad.any():
        ratio = float((d / np.maximum(tol, 1e-300)).max())
        raise AssertionError(f"{what}: {int(bad.sum())} elements beyond tolerance "
                             f"(max abs diff {d.max():.3e}, max diff/tol {ratio:.2f})")


def assert_rel_scaled(got, want, scale, what, rel=REL):
    d = np.abs(np.asarray(got, np.float64) - np.asarray(want, np.float64))
    _report(d, rel * np.asarray(scale, np.float64), what)


def assert_normwise(got, want, what, rel=REL):
    want = np.asarray(want, np.float64)
    d = np.abs(np.asarray(got, np.float64) - want)
    _report(d, np.full_like(d, rel * (np.abs(want).max() if want.size else 0.0)), what)


def update_terms(U, C, V, z_coef_abs=0.0):
    """(T, TZ) of an update U C V^T: T = |U| |C| |V|^T (magnitude of the summed terms),
    TZ = z_coef_abs * NORMAL_ABS * rowsum|U| rowsum|V|^T, with z_coef_abs = eps sum_k |c_k|
    the weight of the Gaussians inside C."""
    U = np.abs(np.asarray(U, np.float64))
    V = np.abs(np.asarray(V, np.float64))
    T = U @ (np.abs(np.asarray(C, np.float64)) @ V.T)
    TZ = z_coef_abs * NORMAL_ABS * np.outer(U.sum(axis=1), V.sum(axis=1))
    return T, TZ


def assert_weights(got, want, dtype, what, before=None, terms=None):
    """bf16: |d| <= 1 bf16 ulp at the operand scale; fp32: relative 1e-5 of it
    (plus the Gaussian allowance TZ).  Returns the number of elements that differ."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    scale = np.abs(want)
    if before is not None:
        scale = np.maximum(scale, np.abs(before))
    extra = 0.0
    if terms is not None:
        scale = np.maximum(scale, terms[0])
        extra = terms[1]
    d = np.abs(got - want)
    if dtype == "bf16":
        _report(d, rounding.bf16_ulp(scale) + extra, what)
    else:
        _report(d, REL * scale + extra, what)
    return int((d > 0).sum())


def gabs(seed, gidx, t, r, rho):
    """(1/q) sum_k |rho_k| |Z_k|: the magnitude of the terms summed into G."""
    acc = np.zeros((r, r))
    for k, rk in enumerate(rho):
        acc += abs(rk) * np.abs(rng.gen_Z(seed, gidx, t, k, r))
    return acc / len(rho)


def assert_moments(M, Vm, M_want, Vm_want, M_prev, Vm_prev, Gabs, beta1, beta2, what):
    assert_rel_scaled(M, M_want, beta1 * np.abs(M_prev) + (1 - beta1) * Gabs, f"M {what}")
    assert_rel_scaled(Vm, Vm_want, beta2 * np.abs(Vm_prev) + (1 - beta2) * Gabs ** 2, f"Vm {what}")

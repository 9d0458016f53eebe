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


# Running totals of the weight comparisons (printed at the end of a pytest session by
# conftest.py): elements compared, elements that differ from the oracle at all, and
# elements within the bound at the operand scale but NOT within it at the result's own
# scale |W_oracle| (plus the Gaussian allowance) -- the ones that pass only because the
# scale was widened to |W_before| or T.
WEIGHT_TOTALS = {"compared": 0, "differ": 0, "widened_only": 0}


def assert_weights(got, want, dtype, what, before=None, terms=None):
    """bf16: |d| <= 1 bf16 ulp at the operand scale; fp32: relative 1e-5 of it
    (plus the Gaussian allowance TZ).  Returns the number of elements that differ."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    strict = np.abs(want)
    scale = strict
    if before is not None:
        scale = np.maximum(scale, np.abs(before))
    extra = 0.0
    if terms is not None:
        scale = np.maximum(scale, terms[0])
        extra = terms[1]
    d = np.abs(got - want)
    if dtype == "bf16":
        tol, tol_strict = rounding.bf16_ulp(scale) + extra, rounding.bf16_ulp(strict) + extra
    else:
        tol, tol_strict = REL * scale + extra, REL * strict + extra
    _report(d, tol, what)
    WEIGHT_TOTALS["compared"] += d.size
    WEIGHT_TOTALS["differ"] += int((d > 0).sum())
    WEIGHT_TOTALS["widened_only"] += int((d > tol_strict).sum())
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


# ----------------------------------------------------------------------------
# Rounding flips of bf16 trajectories, bounded from the arithmetic (not measured)
# ----------------------------------------------------------------------------
# A weight pass computes x = W + delta, delta = U C V^T, with some evaluation error, and
# rounds x once to bf16.  Where the exact x (the oracle's) lies closer to a bf16 rounding
# boundary than the evaluation error can reach, the two sides round to neighbouring values.
# The bounds below are first-order worst-case bounds of each path's fp32 arithmetic, in
# units u = 2^-24, with T = |U| |C| |V|^T (P = C V^T, |P| <= |C| |V|^T elementwise):
#
#   FMA path: P_kj by r fmaf, delta_ij by r fmaf, then W + delta and the bf16 rounding:
#             |d delta| <= 2 r u T (two gamma_r chains) -> c = 2 r + 2, plus u |x|.
#   tensor cores: every operand (V, C in the projection; U, P in the pass) is a scaled fp16
#             pair hi + lo with |x - hi - lo| <= 2^-22 |x| = 4 u |x|; each product drops
#             lo.lo (<= 4 u); each of the k = 3 r / 16 MMAs adds its 16 exact products to
#             the fp32 accumulator with an error taken as <= 2 u of the magnitudes summed
#             (a rounding toward zero allowed).  Projection: (4 + 4 + 4 + 2k) u, then P's
#             own pair 4 u; pass: (4 + 4 + 2k) u; so c = 24 + 4 k, plus u |x| (the fp32
#             multiply-add of the epilogue).
#   C: the coefficient kernel's roundings and the fp32-vs-fp64 Gaussians (NORMAL_ABS), and
#      for the Adam step the propagated error of the fp32 moments (adam_error).
U24 = 2.0 ** -24


def pass_error_coeff(path, r):
    """c of the bound |fl(x) - x| <= (c T + |x|) 2^-24 + |U| dC |V|^T of one weight pass."""
    if path == "fma":
        return 2 * r + 2
    if path == "tc":
        return 24 + 4 * (3 * r // 16)
    raise ValueError(path)


def bf16_boundary_distance(x):
    """Distance of each exact value x to the nearest bf16 rounding boundary (a midpoint
    between the two bf16 values around x): how far an evaluation error has to move x for
    rnd_bf16 to give a neighbouring value."""
    x = np.asarray(x, np.float64)
    ax = np.abs(x)
    y = np.abs(rounding.round_to_bf16(x))
    bits = y.astype(np.float32).view(np.uint32).astype(np.int64)
    up = (bits + 0x10000).astype(np.uint32).view(np.float32).astype(np.float64)
    dn = np.where(bits >= 0x10000,
                  (np.maximum(bits, 0x10000) - 0x10000).astype(np.uint32).view(np.float32)
                  .astype(np.float64), -up)
    return np.minimum((y + up) / 2 - ax, ax - (y + dn) / 2)


def adam_error(dM, dV, M_prev, V_prev, G, dG, M, V, D, beta1, beta2, eps_adam, adam_t):
    """First-order bounds (dM, dV, dD) on the fp32 moments and direction of one subspace
    Adam step (Eqs. (7)-(10)) in the coefficient kernel's order: m = b1 m + a1 g,
    v = b2 v + a2 g^2, D = (m ib1) / (sqrt(v ib2) + eps_adam), ib = fp32(1 / (1 - b^t)),
    given bounds dM, dV on the previous moments and dG on G."""
    b1, b2 = float(beta1), float(beta2)
    a1, a2 = 1.0 - b1, 1.0 - b2
    dM = b1 * dM + a1 * dG + 2 * U24 * (b1 * np.abs(M_prev) + a1 * np.abs(G))
    dV = b2 * dV + a2 * (2 * np.abs(G) * dG + dG ** 2) + 3 * U24 * (b2 * V_prev + a2 * G * G)
    ib1 = 1.0 / (1.0 - b1 ** int(adam_t))
    ib2 = 1.0 / (1.0 - b2 ** int(adam_t))
    Mh, Vh = M * ib1, V * ib2
    dMh = ib1 * dM + 2 * U24 * np.abs(Mh)
    dVh = ib2 * dV + 2 * U24 * Vh
    s = np.sqrt(Vh)
    ds = np.where(s > 0, dVh / (2 * np.maximum(s, 1e-300)), np.sqrt(dVh)) + U24 * s
    den = s + float(eps_adam)
    dden = ds + U24 * den
    dD = (dMh + np.abs(D) * dden) / den + U24 * np.abs(D)
    return dM, dV, dD


class FlipLedger:
    """Per-element record, along the oracle's trajectory, of the passes whose exact value
    lies within the evaluation-error bound E of a bf16 rounding boundary ("ambiguous"),
    and of the probability that the computed trajectory ends on a different value when
    each pass's error is uniform on [-E, E] (a flip at distance d < E then has
    probability (E - d) / 2E)."""

    def __init__(self, shape):
        self.n_amb = np.zeros(shape, np.int64)
        self.log_keep = np.zeros(shape)

    def record(self, x, E):
        d = bf16_boundary_distance(x)
        self.n_amb += d < E
        p = np.clip((E - d) / (2 * np.maximum(E, 1e-300)), 0.0, 0.5)
        self.log_keep += np.log1p(-p)

    def flip_probability(self):
        return -np.expm1(self.log_keep)


def bounded_pass(W, U, V, C, dC, path, r, ledger):
    """One bf16 weight pass of the oracle (x = W + U C V^T exact, rounded once) that also
    records x and its error bound in the ledger.  dC: elementwise bound on C's error."""
    from oracle import subzero
    x = np.asarray(W, np.float64) + subzero.delta(U, V, C)
    aU, aV = np.abs(U), np.abs(V)
    T = aU @ (np.abs(C) @ aV.T)
    E = (pass_error_coeff(path, r) * T + np.abs(x)) * U24 + aU @ (dC @ aV.T)
    ledger.record(x, E)
    return rounding.round_to_bf16(x)

"""The parity helpers' tolerances, checked on the CPU (no GPU).

The GPU tests accept a result when tests/parity.py's bounds hold.  Here simulated
kernel outputs, made from the oracle's own definitions, show that those bounds accept
what a correct fp32 evaluation produces (fp32 products and sums, rounding through fp32,
fp32 Gaussians within their stated allowance) and reject the mistakes a kernel could
plausibly make (a dropped rank-r term, a flipped sign, the wrong query's Z, a transposed
coefficient, an element off by twice its bound, a moment missing its (1 - beta) or its
square).
"""

import numpy as np
import pytest

from oracle import haar, rng, rounding, subzero
from parity import NORMAL_ABS, assert_moments, assert_weights, gabs, update_terms

SEED, M_, N_, R_ = 31, 96, 80, 8


def _case(dtype, eps):
    U, V = haar.haar_proj(SEED, 0, 0, M_, N_, R_)
    W = np.random.default_rng(2).standard_normal((M_, N_)) * 0.02
    W = rounding.round_to(W, dtype)
    C = subzero.perturb_coeff(SEED, 0, 0, R_, [(0, 1.0), (1, -1.0)], eps)
    want = subzero.apply_pass(W, dtype, U, V, C)
    terms = update_terms(U, C, V, z_coef_abs=2 * eps)
    return U, V, W, C, want, terms


def _fp32_pass(W, U, V, C, dtype):
    """W + U (C V^T) evaluated in fp32 (products and sums), rounded through fp32."""
    f = np.float32
    P = C.astype(f) @ V.astype(f).T
    d = U.astype(f) @ P
    return rounding.round_to((W.astype(f) + d).astype(np.float64), dtype)


@pytest.mark.parametrize("dtype,eps", [("bf16", 1e-3), ("bf16", 1e-1), ("f32", 1e-3), ("f32", 1e-1)])
def test_a_correct_fp32_evaluation_passes(dtype, eps):
    U, V, W, C, want, terms = _case(dtype, eps)
    assert_weights(_fp32_pass(W, U, V, C, dtype), want, dtype, "fp32 evaluation",
                   before=W, terms=terms)
    # the Gaussians drawn in fp32: each entry of Z off by up to the stated allowance
    dz = np.random.default_rng(3).uniform(-NORMAL_ABS, NORMAL_ABS, (R_, R_))
    C_gpu = C + 2 * eps * dz / 2          # two terms, |c_k| = 1 each, half the allowance apiece
    assert_weights(_fp32_pass(W, U, V, C_gpu, dtype), want, dtype, "fp32 Gaussians",
                   before=W, terms=terms)


def _mistakes(U, V, W, C, dtype, eps, terms):
    Z1 = rng.gen_Z(SEED, 0, 0, 1, R_)
    Z2 = rng.gen_Z(SEED, 0, 0, 2, R_)
    off = subzero.apply_pass(W, dtype, U, V, C)
    off2 = off.copy()
    # one element moved by twice its bound: one ulp (bf16) or 1e-5 (fp32) of the operand
    # scale max(|W_new|, |W_before|, T), plus the Gaussian allowance
    i, j = 7, 11
    scale = max(abs(off2[i, j]), abs(W[i, j]), terms[0][i, j])
    bound = (rounding.bf16_ulp(scale) if dtype == "bf16" else 1e-5 * scale) + terms[1][i, j]
    off2[i, j] += 2 * bound
    return {
        "dropped rank term": rounding.round_to(W + U[:, :-1] @ (C @ V.T)[:-1], dtype),
        "flipped sign": subzero.apply_pass(W, dtype, U, V, -C),
        "wrong query": subzero.apply_pass(W, dtype, U, V, eps * (rng.gen_Z(SEED, 0, 0, 0, R_) - Z2)),
        "transposed C": subzero.apply_pass(W, dtype, U, V, C.T),
        "one element off": off2,
        "no update": W.copy(),
        "query 1 only": subzero.apply_pass(W, dtype, U, V, -eps * Z1),
    }


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_plausible_kernel_mistakes_are_rejected(dtype):
    eps = 1e-1                                  # the stress setting the parity tests also run
    U, V, W, C, want, terms = _case(dtype, eps)
    for name, got in _mistakes(U, V, W, C, dtype, eps, terms).items():
        with pytest.raises(AssertionError):
            assert_weights(got, want, dtype, name, before=W, terms=terms)


def test_moment_tolerance_accepts_fp32_and_rejects_mistakes():
    r, q, b1, b2 = R_, 4, 0.9, 0.95
    rho = np.array([3.0, -1.5, 0.25, 2.0])
    G = subzero.grad_G(SEED, 0, 0, r, rho)
    rs = np.random.default_rng(5)
    M0, V0 = rs.standard_normal((r, r)) * 0.1, np.abs(rs.standard_normal((r, r))) * 0.1
    M, Vm, _, _, _ = subzero.adam(M0, V0, G, b1, b2, 1e-8, 3)
    Gabs = gabs(SEED, 0, 0, r, rho)
    f = np.float32
    G32 = sum(f(rho[k]) * rng.gen_Z(SEED, 0, 0, k, r).astype(f) for k in range(q)) / f(q)
    M32 = f(b1) * M0.astype(f) + f(1 - b1) * G32
    V32 = f(b2) * V0.astype(f) + f(1 - b2) * G32 * G32
    assert_moments(M32, V32, M, Vm, M0, V0, Gabs, b1, b2, "fp32")
    bad = {
        "M without (1 - beta1)": (b1 * M0 + G, Vm),
        "Vm from G, not G*G": (M, b2 * V0 + (1 - b2) * G),
        "betas swapped": (b2 * M0 + (1 - b2) * G, b1 * V0 + (1 - b1) * G * G),
        "G without 1/q": (b1 * M0 + (1 - b1) * q * G, Vm),
    }
    for name, (Mb, Vb) in bad.items():
        with pytest.raises(AssertionError):
            assert_moments(Mb, Vb, M, Vm, M0, V0, Gabs, b1, b2, name)

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


# ---------------------------------------------------------------------------------------
# The flip bounds of the bf16 trajectory test (parity.pass_error_coeff / FlipLedger)
# ---------------------------------------------------------------------------------------

def _fma_chain(a, b):
    """sum_k a[:, k] b[k, :] by one fmaf per term in k order (fp32, each fma rounded once;
    the exact product-plus-accumulator is formed in fp64 first)."""
    acc = np.zeros((a.shape[0], b.shape[1]), np.float32)
    for k in range(a.shape[1]):
        acc = (np.outer(a[:, k].astype(np.float64), b[k].astype(np.float64)) + acc).astype(np.float32)
    return acc


def _sim_fma_pass(W, U, V, C):
    """The FMA path's arithmetic: P = C V^T and U P by fmaf chains, W + delta in fp32."""
    f = np.float32
    P = _fma_chain(C.astype(f), V.astype(f).T)
    d = _fma_chain(U.astype(f), P)
    return (W.astype(f) + d).astype(np.float64)


def _pair16(x, s):
    """Scaled fp16 pair: x s = hi + lo (RNE, subnormals kept)."""
    xs = (np.asarray(x, np.float32) * np.float32(s)).astype(np.float32)
    hi = xs.astype(np.float16)
    lo = (xs - hi.astype(np.float32)).astype(np.float16)
    return hi.astype(np.float64), lo.astype(np.float64)


def _mma_chain(ah, al, bh, bl):
    """hi.hi + hi.lo + lo.hi over K in MMAs of 16: each MMA's 16 exact products are added
    to the fp32 accumulator with one rounding (the kernels' order: K chunk by K chunk, the
    three products of a chunk in turn)."""
    K = ah.shape[1]
    acc = np.zeros((ah.shape[0], bh.shape[1]), np.float32)
    for k0 in range(0, K, 16):
        sl = slice(k0, k0 + 16)
        for x, y in ((ah, bh), (ah, bl), (al, bh)):
            acc = (x[:, sl] @ y[sl] + acc.astype(np.float64)).astype(np.float32)
    return acc


def _sim_tc_pass(W, U, V, C, r, scale_err=1.0):
    """The tensor-core path's arithmetic with the scales of zo_tc_common.cuh: V, C, U, P as
    fp16 pairs (V, U at 2^14, C at 2^(14 - E), max|C| < 2^E, P at 2^(e_C + off(r))), three
    products per K chunk into fp32, the epilogue's fp32 multiply-add.  scale_err != 1
    plants a mistake: the P pair formed at a scale off by that factor but undone as if not."""
    off = -1 if r <= 16 else -2 if r <= 64 else -3
    e_c = 14 - int(np.frexp(np.abs(C).max())[1])
    vh, vl = _pair16(V, 2.0 ** 14)
    ch, cl = _pair16(C, 2.0 ** e_c)
    D = _mma_chain(vh, vl, ch.T, cl.T)                     # (V C^T) 2^(14 + e_C) = P^T s
    e_p = e_c + off
    Pt = (D.astype(np.float64) * 2.0 ** (off - 14)).astype(np.float32)
    ph, pl = _pair16(Pt.T, scale_err)
    uh, ul = _pair16(U, 2.0 ** 14)
    acc = _mma_chain(uh, ul, ph, pl)
    w = np.float32(2.0 ** (-14 - e_p))
    return (acc.astype(np.float64) * w + W.astype(np.float32).astype(np.float64)).astype(np.float32) \
        .astype(np.float64)


@pytest.mark.parametrize("path,r", [("fma", 8), ("fma", 32), ("tc", 16), ("tc", 32), ("tc", 64)])
@pytest.mark.parametrize("eps", [1e-3, 1e-1, 1.0])
def test_flip_bound_covers_the_simulated_arithmetic(path, r, eps):
    # every element whose simulated rounding differs from the exact one has its exact value
    # within the derived error bound of a rounding boundary
    from parity import FlipLedger, bounded_pass
    m, n = 160, 136
    U, V = haar.haar_proj(SEED, 3, 0, m, n, r)
    U, V = U.astype(np.float32).astype(np.float64), V.astype(np.float32).astype(np.float64)
    W = rounding.round_to_bf16(np.random.default_rng(r).standard_normal((m, n)) * 0.02)
    flips = near = 0
    for k in range(4):
        C = subzero.perturb_coeff(SEED, 3, k, r, [(0, 1.0), (1, -1.0)], eps)
        C = C.astype(np.float32).astype(np.float64)          # the C the kernels hold
        ledger = FlipLedger(W.shape)
        want = bounded_pass(W, U, V, C, np.zeros_like(C), path, r, ledger)
        x = _sim_fma_pass(W, U, V, C) if path == "fma" else _sim_tc_pass(W, U, V, C, r)
        differ = rounding.round_to_bf16(x) != want
        assert not (differ & (ledger.n_amb == 0)).any()
        flips += int(differ.sum())
        near += int((ledger.n_amb > 0).sum())
    assert near >= flips


def test_flip_bound_rejects_a_pair_at_the_wrong_scale():
    # a P pair formed at twice the scale the epilogue undoes doubles delta: nearly every
    # element rounds differently, far outside the bound
    from parity import FlipLedger, bounded_pass
    m, n, r = 160, 136, 32
    U, V = haar.haar_proj(SEED, 4, 0, m, n, r)
    W = rounding.round_to_bf16(np.random.default_rng(5).standard_normal((m, n)) * 0.02)
    C = subzero.perturb_coeff(SEED, 4, 0, r, [(0, 1.0)], 1e-1).astype(np.float32).astype(np.float64)
    ledger = FlipLedger(W.shape)
    want = bounded_pass(W, U, V, C, np.zeros_like(C), "tc", r, ledger)
    x = _sim_tc_pass(W, U, V, C, r, scale_err=2.0)
    differ = rounding.round_to_bf16(x) != want
    assert (differ & (ledger.n_amb == 0)).sum() > differ.size // 4


def test_boundary_distance_is_the_rounding_margin():
    from parity import bf16_boundary_distance
    x = np.random.default_rng(7).standard_normal(20000) * 0.02
    x = np.concatenate([x, [1.0, -1.0, 2.0 ** -3, 3.0 * 2.0 ** -9]])   # values on a binade edge
    d = bf16_boundary_distance(x)
    r0 = rounding.round_to_bf16(x)
    s = np.sign(x)
    assert (d >= 0).all()
    # just inside the margin the rounding holds on both sides; just past it, on one side, it
    # changes
    assert (rounding.round_to_bf16(x + d * (1 - 1e-6)) == r0).all()
    assert (rounding.round_to_bf16(x - d * (1 - 1e-6)) == r0).all()
    moved = (rounding.round_to_bf16(x + s * d * (1 + 1e-6)) != r0) | \
            (rounding.round_to_bf16(x - s * d * (1 + 1e-6)) != r0)
    assert moved.all()

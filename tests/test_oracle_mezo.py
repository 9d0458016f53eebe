"""Pins of the oracle's full-space SPSA perturbation (Eq. (1)) (no GPU)."""

import numpy as np
from scipy import stats

from oracle import mezo, rng, rounding


def test_row_streams_follow_the_counter_contract():
    # row 3 of a 10-column matrix uses counter words 3*3 .. 3*3+2, lanes in order
    seed, i, t, n = 77, 5, 9, 10
    z = mezo.gen_full_z(seed, i, t, n, [3])[0]
    words = rng.philox4x32_10(
        np.array([[9 + k, i, t, 5 << 24] for k in range(3)], np.uint64),
        np.array([[77, 0]] * 3, np.uint64)).reshape(-1)
    u = rng.uniform_from_u32(words).reshape(-1, 4)
    rad = np.sqrt(-2 * np.log(u[:, 0]))
    assert np.allclose(z[0::4][:3], rad * np.cos(2 * np.pi * u[:, 1]), atol=1e-15)
    assert np.allclose(z[1::4][:3], rad * np.sin(2 * np.pi * u[:, 1]), atol=1e-15)
    # rows are independent of how many rows are drawn together
    both = mezo.gen_full_z(seed, i, t, n, [1, 3])
    assert np.array_equal(both[1], z)


def test_full_z_is_standard_normal_and_uncorrelated_across_steps():
    a = mezo.gen_full_z(1, 0, 0, 1000, np.arange(300)).ravel()
    b = mezo.gen_full_z(1, 0, 1, 1000, np.arange(300)).ravel()
    assert stats.kstest(a, "norm").pvalue > 1e-3
    assert abs(np.corrcoef(a, b)[0, 1]) < 5 / np.sqrt(a.size)


def test_perturb_restore_is_exact_in_fp64_and_rounds_once():
    W = np.random.default_rng(0).standard_normal((20, 37)) * 0.02
    eps = 1e-3
    Wp = mezo.mezo_pass(W, "f64", 3, 1, 2, eps)
    Wm = mezo.mezo_pass(Wp, "f64", 3, 1, 2, -2 * eps)
    Wr = mezo.mezo_pass(Wm, "f64", 3, 1, 2, eps)
    assert np.max(np.abs(Wr - W)) < 1e-16
    Z = mezo.gen_full_z(3, 1, 2, 37, np.arange(20))
    Wb = rounding.round_to_bf16(W)
    assert np.array_equal(mezo.mezo_pass(Wb, "bf16", 3, 1, 2, 0.1),
                          rounding.round_to_bf16(Wb + 0.1 * Z))
    assert np.array_equal(mezo.mezo_pass(Wb[[2, 7]], "bf16", 3, 1, 2, 0.1, rows=[2, 7]),
                          rounding.round_to_bf16(Wb + 0.1 * Z)[[2, 7]])


def test_spsa_scalar_is_the_directional_derivative_of_a_quadratic():
    # Eq. (1): for L(w) = 1/2 |w|^2 the central difference is exactly <w, z>
    rs = np.random.default_rng(4)
    w, z, eps = rs.standard_normal(50), rs.standard_normal(50), 1e-2
    L = lambda v: 0.5 * v @ v
    assert abs(mezo.spsa_rho(L(w + eps * z), L(w - eps * z), eps) - w @ z) < 1e-12

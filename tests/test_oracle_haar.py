"""Pins of the oracle's Alg. 1 (QR + sign correction) (no GPU)."""

import numpy as np
import pytest
from scipy import stats

from oracle import haar, rng

SHAPES = [(4, 4), (8, 4), (50, 10), (256, 8), (300, 32), (1000, 64), (5120, 4)]


@pytest.mark.parametrize("m,r", SHAPES)
def test_householder_factorises(m, r):
    A = rng.gen_omega(11, m, r, "U", m, r)
    Q, R = haar.householder_qr(A)
    assert np.allclose(Q.T @ Q, np.eye(r), rtol=0, atol=1e-12)
    assert np.allclose(Q @ R, A, rtol=0, atol=1e-10 * max(1.0, np.abs(A).max()))
    assert np.array_equal(R, np.triu(R))


@pytest.mark.parametrize("m,r", SHAPES)
def test_raw_factors_follow_lapack_convention(m, r):
    # LAPACK's geqrf/orgqr (numpy.linalg.qr) use the same reflector convention,
    # so even the unnormalised factors agree.
    A = rng.gen_omega(12, m, r, "V", m, r)
    Q, R = haar.householder_qr(A)
    Ql, Rl = np.linalg.qr(A, mode="reduced")
    assert np.allclose(Q, Ql, rtol=0, atol=1e-11)
    assert np.allclose(R, Rl, rtol=0, atol=1e-10 * np.abs(Rl).max())


@pytest.mark.parametrize("m,r", SHAPES)
def test_sign_corrected_factor_is_the_unique_positive_diagonal_qr(m, r):
    A = rng.gen_omega(13, m, r, "U", m, r)
    Q, R = haar.haar_from_gaussian(A)
    assert np.all(np.diag(R) > 0)
    assert np.allclose(Q @ R, A, rtol=0, atol=1e-10 * max(1.0, np.abs(A).max()))
    # Cholesky definition: R = chol(A^T A)^T, Q = A R^{-1}
    L = np.linalg.cholesky(A.T @ A)
    Qc = np.linalg.solve(L, A.T).T
    assert np.allclose(Q, Qc, rtol=0, atol=1e-9)
    assert np.allclose(R, L.T, rtol=0, atol=1e-9 * np.abs(R).max())
    # and LAPACK's QR followed by the same sign rule lands on the same factor
    Ql, Rl = np.linalg.qr(A, mode="reduced")
    s = np.where(np.diag(Rl) < 0, -1.0, 1.0)
    assert np.allclose(Q, Ql * s, rtol=0, atol=1e-11)


def test_sign_correction_handles_zero_diagonal_as_plus_one():
    A = np.array([[0.0, 1.0], [0.0, 2.0], [0.0, 0.0]])
    A[:, 0] = 0.0
    Q, R = haar.householder_qr(A)
    Qs, Rs = haar.sign_correct(Q, R)
    assert Rs[0, 0] == 0.0 and np.allclose(Qs[:, 0], Q[:, 0])


def test_haar_m2_r1_angle_is_uniform_on_the_full_circle():
    # For m = 2, r = 1 the Haar column is uniform on the unit circle.  Raw
    # LAPACK-convention QR only covers the half circle opposite to sign(x_0).
    ang, raw_ang = [], []
    for j in range(4000):
        om = rng.gen_omega(21, 0, j, "U", 2, 1)
        Q, R = haar.householder_qr(om)
        Qs, _ = haar.sign_correct(Q, R)
        ang.append(np.arctan2(Qs[1, 0], Qs[0, 0]) % (2 * np.pi))
        raw_ang.append(np.arctan2(Q[1, 0], Q[0, 0]) % (2 * np.pi))
    assert stats.kstest(np.array(ang) / (2 * np.pi), "uniform").pvalue > 1e-3
    assert stats.kstest(np.array(raw_ang) / (2 * np.pi), "uniform").pvalue < 1e-6


def test_haar_moments_on_small_shapes():
    # E[Q_ij^2] = 1/m, E[Q_ij^4] = 3/(m(m+2)), E[Q_i1 Q_j1] = 0 (i != j)
    m, r, trials = 5, 2, 4000
    Qs = np.stack([haar.haar_proj(31, 0, j, m, 3, r)[0] for j in range(trials)])
    q2 = (Qs ** 2).mean(axis=0)
    q4 = (Qs ** 4).mean(axis=0)
    se2 = np.sqrt((3 / (m * (m + 2)) - 1 / m ** 2) / trials)
    assert np.all(np.abs(q2 - 1 / m) < 5 * se2)
    assert np.all(np.abs(q4 - 3 / (m * (m + 2))) < 0.1 * 3 / (m * (m + 2)))
    cross = (Qs[:, 0, 0] * Qs[:, 1, 0]).mean()
    assert abs(cross) < 5 * np.sqrt(1 / (m * (m + 2)) / trials)


def test_paper_protocol_ks_against_normalised_gaussian():
    # App. A.3: m = 50, r = 10, 2000 trials, one coordinate of the first column
    # of Q against normalised Gaussian vectors (uniform on S^(m-1)).
    m, r, trials = 50, 10, 2000
    corrected, raw, ref = [], [], []
    for j in range(trials):
        om = rng.gen_omega(0, 7, j, "U", m, r)
        Q, R = haar.householder_qr(om)
        Qs, _ = haar.sign_correct(Q, R)
        corrected.append(Qs[0, 0])
        raw.append(Q[0, 0])
        g = rng.normals(0, 8, j, 0, m)
        ref.append(g[0] / np.linalg.norm(g))
    corrected, raw, ref = map(np.asarray, (corrected, raw, ref))
    assert stats.ks_2samp(corrected, ref).pvalue > 0.01
    assert stats.ks_2samp(raw, ref).pvalue < 1e-3
    # coordinate variance 1/m (App. A.3 quotes the theoretical 0.02)
    assert abs(corrected.var() - 1 / m) < 5 * np.sqrt(2 / trials) / m

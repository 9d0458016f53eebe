"""Alg. 1 (Haar-distributed projection bases) of the oracle (test infrastructure only).

Sec. 4.3 / Eq. (11): draw a Gaussian Omega (rows x r), take its thin QR
Omega = Q~ R~, and multiply column j of Q~ by sgn(R~_jj).  The result is the
unique thin QR factor whose triangular factor has a positive diagonal, which
is Haar-distributed (Mezzadri 2007; App. A.3 validates it empirically).

The QR itself is textbook Householder (Golub & Van Loan, Matrix Computations,
Sec. 5.1-5.2) in the LAPACK reflector convention: for the column x = A[j:, j],
beta = -sign(x_0) ||x||, v = x / (x_0 - beta) with v_0 = 1,
tau = (beta - x_0) / beta, and H_j = I - tau v v^T maps x to beta e_1.  This
convention can leave R~_jj negative, which is exactly the ambiguity Eq. (11)
removes.  sgn(0) is read as +1 (a measure-zero event for Gaussian input).
"""

import math

import numpy as np

from . import rng


def householder_qr(A):
    """Thin QR of A (m x r, m >= r) by Householder reflections, fp64.

    Returns (Q, R): Q is m x r with orthonormal columns, R is r x r upper
    triangular, A = Q R.  No sign normalisation (R's diagonal may be negative).
    """
    A = np.array(A, dtype=np.float64, copy=True)
    m, r = A.shape
    if m < r:
        raise ValueError("thin QR needs rows >= columns")
    taus = np.zeros(r)
    for j in range(r):
        x = A[j:, j]
        alpha = x[0]
        sigma = float(x[1:] @ x[1:])
        if sigma == 0.0:
            tau, beta = 0.0, alpha
            v = np.zeros_like(x)
            v[0] = 1.0
        else:
            beta = -math.copysign(math.sqrt(alpha * alpha + sigma), alpha)
            tau = (beta - alpha) / beta
            v = x / (alpha - beta)
            v[0] = 1.0
        # apply H_j to the trailing columns
        if j + 1 < r:
            w = v @ A[j:, j + 1:]
            A[j:, j + 1:] -= tau * np.outer(v, w)
        A[j, j] = beta
        A[j + 1:, j] = v[1:]
        taus[j] = tau
    R = np.triu(A[:r, :])
    # thin Q = H_0 H_1 ... H_{r-1} [I_r; 0], accumulated from the last reflector
    Q = np.zeros((m, r))
    Q[:r, :r] = np.eye(r)
    for j in reversed(range(r)):
        v = np.concatenate(([1.0], A[j + 1:, j]))
        w = v @ Q[j:, :]
        Q[j:, :] -= taus[j] * np.outer(v, w)
    return Q, R


def sign_correct(Q, R):
    """Eq. (11): Q <- Q diag(sgn R_jj), R <- diag(sgn R_jj) R (sgn(0) = +1)."""
    d = np.diag(R)
    s = np.where(d < 0.0, -1.0, 1.0)
    return Q * s[None, :], R * s[:, None]


def haar_from_gaussian(omega):
    """Alg. 1 on a given Gaussian matrix: QR then the sign correction."""
    Q, R = householder_qr(omega)
    return sign_correct(Q, R)


def haar_proj(seed, i, j, m, n, r):
    """Alg. 1 for matrix i (m_i x r and n_i x r bases) at refresh j.

    Omega_U (m x r) and Omega_V (n x r) come from the counter contract of
    ``oracle.rng`` (tags 2 and 3).  Returns (U, V), both fp64.
    """
    om_u = rng.gen_omega(seed, i, j, "U", m, r)
    om_v = rng.gen_omega(seed, i, j, "V", n, r)
    U, _ = haar_from_gaussian(om_u)
    V, _ = haar_from_gaussian(om_v)
    return U, V

"""Pins of the oracle's perturbed linear layer (oracle/subzero.py: perturbed_linear).

Y = X (W + U C V^T)^T is the output of one linear layer of the loss evaluation of Alg. 3
at the perturbed weights (Eq. (4) form), with W itself left untouched.  The pins do not
re-type the oracle's formula: a hand-computed case, brute-force loops over the scalar
definition, the factorised order X W^T + ((X V) C^T) U^T in which the CUDA path sums it,
linearity in C, and the weight-pass oracle at the same coefficient.
"""

import numpy as np
import pytest

from oracle import rounding, subzero


def test_hand_computed_1x2x2(golden):
    rows = {r[0]: np.array([float(x) for x in r[1:]]) for r in golden("perturbed_linear_1x2x2.txt")}
    X = rows["X"].reshape(1, 2)
    W = rows["W"].reshape(2, 2)
    U = rows["U"].reshape(2, 1)
    V = rows["V"].reshape(2, 1)
    C = rows["C"].reshape(1, 1)
    Y = subzero.perturbed_linear(X, W, U, V, C, "f64")
    assert np.array_equal(Y, rows["Y"].reshape(1, 2))


def _brute(X, W, U, V, C):
    T, n = len(X), len(X[0])
    m, r = len(U), len(U[0])
    Y = [[0.0] * m for _ in range(T)]
    for t in range(T):
        for o in range(m):
            acc = 0.0
            for j in range(n):
                w = W[o][j]
                for a in range(r):
                    for b in range(r):
                        w += U[o][a] * C[a][b] * V[j][b]
                acc += X[t][j] * w
            Y[t][o] = acc
    return np.array(Y)


@pytest.mark.parametrize("T,n,m,r", [(3, 5, 4, 2), (2, 7, 3, 3), (1, 4, 6, 4)])
def test_brute_force_definition(T, n, m, r):
    rs = np.random.default_rng(T * 100 + n * 10 + m + r)
    X, W = rs.standard_normal((T, n)), rs.standard_normal((m, n))
    U, V, C = rs.standard_normal((m, r)), rs.standard_normal((n, r)), rs.standard_normal((r, r))
    got = subzero.perturbed_linear(X, W, U, V, C, "f64")
    want = _brute(X.tolist(), W.tolist(), U.tolist(), V.tolist(), C.tolist())
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)


def test_factorised_order_and_linearity_in_C():
    rs = np.random.default_rng(7)
    T, n, m, r = 9, 40, 24, 8
    X, W = rs.standard_normal((T, n)), rs.standard_normal((m, n))
    U, V = rs.standard_normal((m, r)), rs.standard_normal((n, r))
    C1, C2 = rs.standard_normal((r, r)), rs.standard_normal((r, r))
    f = lambda C: subzero.perturbed_linear(X, W, U, V, C, "f64")   # noqa: E731
    # the order the CUDA path uses: the dense product plus a rank-r term, S = (X V) C^T
    S = (X @ V) @ C1.T
    assert np.allclose(f(C1), X @ W.T + S @ U.T, rtol=1e-12, atol=1e-10)
    # a transposed C would give (X V) C U^T instead: the two differ for a generic C
    assert not np.allclose(f(C1), X @ W.T + ((X @ V) @ C1) @ U.T, rtol=1e-6)
    assert np.allclose(f(C1 + C2) - f(C1) - f(C2) + f(np.zeros((r, r))), 0.0, atol=1e-10)


def test_agrees_with_the_weight_pass_oracle():
    # evaluating at the exact perturbed weight equals evaluating at the weight-pass
    # oracle's W + U C V^T kept in fp64; rounding the output once gives bf16 values
    rs = np.random.default_rng(3)
    T, n, m, r = 5, 33, 17, 4
    X = rounding.round_to_bf16(rs.standard_normal((T, n)))
    W = rounding.round_to_bf16(0.02 * rs.standard_normal((m, n)))
    U, V = np.linalg.qr(rs.standard_normal((m, r)))[0], np.linalg.qr(rs.standard_normal((n, r)))[0]
    C = 1e-3 * subzero.perturb_coeff(11, 2, 0, r, [(0, 1.0), (1, -1.0)], 1.0)
    Wp = subzero.apply_pass(W, "f64", U, V, C)
    assert np.allclose(subzero.perturbed_linear(X, W, U, V, C, "f64"), X @ Wp.T, rtol=1e-13,
                       atol=1e-15)
    Y = subzero.perturbed_linear(X, W, U, V, C, "bf16")
    assert np.array_equal(Y, rounding.round_to_bf16(Y))

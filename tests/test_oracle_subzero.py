"""Pins of the oracle's perturbation, estimator, subspace Adam and schedule (no GPU)."""

import numpy as np
import pytest

from oracle import haar, rng, rounding, subzero


def _basis(m, n, r, seed=3, j=0):
    return haar.haar_proj(seed, 0, j, m, n, r)


@pytest.mark.parametrize("m,n,r", [(16, 12, 4), (64, 40, 8), (300, 200, 16)])
def test_lemma1_isometry_and_projection(m, n, r):
    # Lemma 1 (Sec. 3): vec(U C V^T) = (V kron U) vec(C) with V kron U
    # column-orthonormal, hence ||U C V^T||_F = ||C||_F and U^T (U C V^T) V = C.
    U, V = _basis(m, n, r)
    C = rng.gen_Z(4, 0, 0, 0, r)
    D = subzero.delta(U, V, C)
    assert abs(np.linalg.norm(D) - np.linalg.norm(C)) < 1e-12 * np.linalg.norm(C)
    assert np.allclose(U.T @ D @ V, C, rtol=0, atol=1e-12)
    # the Kronecker form itself, elementwise, on the small case
    if m * n <= 4096:
        K = np.kron(V, U)
        assert np.allclose(K @ C.flatten(order="F"), D.flatten(order="F"), atol=1e-13)


def test_perturb_then_restore_is_identity_in_exact_arithmetic():
    m, n, r = 40, 30, 8
    U, V = _basis(m, n, r)
    W = np.random.default_rng(0).standard_normal((m, n)) * 0.02
    Cp = subzero.perturb_coeff(1, 0, 0, r, [(0, 1.0)], 1e-3)
    Cm = subzero.perturb_coeff(1, 0, 0, r, [(0, -1.0)], 1e-3)
    W2 = subzero.apply_pass(subzero.apply_pass(W, "f64", U, V, Cp), "f64", U, V, Cm)
    assert np.max(np.abs(W2 - W)) < 1e-15


def test_pass_rounds_once_to_storage_dtype():
    m, n, r = 32, 24, 4
    U, V = _basis(m, n, r)
    W = rounding.round_to_bf16(np.random.default_rng(1).standard_normal((m, n)) * 0.02)
    C = subzero.perturb_coeff(2, 0, 0, r, [(0, 1.0)], 0.1)
    out = subzero.apply_pass(W, "bf16", U, V, C)
    exact = W + U @ C @ V.T
    assert np.array_equal(out, rounding.round_to_bf16(exact))
    assert np.all(np.abs(out - exact) <= rounding.bf16_ulp(out) / 2 * (1 + 1e-12))
    # row subsets give the same rows
    rows = np.array([0, 5, 31])
    assert np.array_equal(subzero.apply_pass(W[rows], "bf16", U, V, C, rows=rows), out[rows])


def test_rho_from_losses_schemes():
    eps = 1e-3
    L = np.array([2.5, 2.25, 1.0, 1.5], np.float32)
    assert np.allclose(subzero.rho_from_losses(L, "central", eps, 2),
                       [0.25 / 2e-3, -0.5 / 2e-3], rtol=1e-15)
    L = np.array([2.0, 2.5, 1.5], np.float32)
    assert np.allclose(subzero.rho_from_losses(L, "forward", eps, 2), [500.0, -500.0], rtol=1e-15)
    assert np.array_equal(subzero.rho_from_losses(np.array([1.0, 2.0]), "direct", eps, 2), [1.0, 2.0])


def test_G_single_query_unit_rho_is_Z_and_is_linear_in_rho():
    r = 6
    G = subzero.grad_G(9, 2, 5, r, np.array([1.0]))
    assert np.array_equal(G, rng.gen_Z(9, 2, 5, 0, r))
    a = np.array([0.3, -1.2, 2.0, 0.7])
    b = np.array([1.5, 0.25, -0.5, 3.0])
    Ga, Gb = subzero.grad_G(9, 2, 5, r, a), subzero.grad_G(9, 2, 5, r, b)
    Gab = subzero.grad_G(9, 2, 5, r, 2 * a - 3 * b)
    assert np.allclose(Gab, 2 * Ga - 3 * Gb, rtol=0, atol=1e-13)
    # 1/q normalisation: q identical queries average to one
    Z = [rng.gen_Z(9, 2, 5, k, r) for k in range(4)]
    assert np.allclose(subzero.grad_G(9, 2, 5, r, np.ones(4)), sum(Z) / 4, atol=1e-15)


def test_adam_hand_computed_2x2(golden):
    rows = {r[0]: np.array([float(x) for x in r[1:]]).reshape(2, 2) for r in golden("adam_2x2.txt")}
    G = rows["G"]
    M, Vm = np.zeros((2, 2)), np.zeros((2, 2))
    M, Vm, D, Mh, Vh = subzero.adam(M, Vm, G, 0.9, 0.999, 1e-8, 1)
    assert np.allclose(M, rows["M1"], rtol=1e-14, atol=0)
    assert np.allclose(Vm, rows["Vm1"], rtol=1e-13, atol=0)
    assert np.allclose(Mh, G, rtol=1e-14) and np.allclose(Vh, G * G, rtol=1e-12)
    assert np.allclose(D, rows["D1"], rtol=1e-13, atol=0)
    M, Vm, D, Mh, Vh = subzero.adam(M, Vm, G, 0.9, 0.999, 1e-8, 2)
    assert np.allclose(M, rows["M2"], rtol=1e-14, atol=0)
    assert np.allclose(Vm, rows["Vm2"], rtol=1e-12, atol=0)
    assert np.allclose(D, rows["D2"], rtol=1e-12, atol=0)


def _net_perturbation(plan_passes):
    """Net coefficient of each Z_k after each pass of a plan."""
    net, out = {}, []
    for terms in plan_passes:
        for k, c in terms:
            net[k] = net.get(k, 0.0) + c
        out.append({k: v for k, v in net.items() if v != 0.0})
    return out


@pytest.mark.parametrize("q", [1, 2, 4, 8])
def test_pass_plans_visit_the_paper_evaluation_points(q):
    # central (Eq. (3)): loss evaluations at W + eps Z_k and W - eps Z_k
    passes, restore = subzero.pass_plan("central", q)
    assert len(passes) == 2 * q
    nets = _net_perturbation(passes)
    for k in range(q):
        assert nets[2 * k] == {k: 1.0} and nets[2 * k + 1] == {k: -1.0}
    final = _net_perturbation(passes + [restore])[-1]
    assert final == {}
    # forward (Alg. 3, Eq. (6)): evaluations at W + eps Z_k
    passes, restore = subzero.pass_plan("forward", q)
    assert len(passes) == q
    nets = _net_perturbation(passes)
    for k in range(q):
        assert nets[k] == {k: 1.0}
    assert _net_perturbation(passes + [restore])[-1] == {}


def test_fused_equals_unfused_in_exact_arithmetic():
    m, n, r, q = 24, 20, 4, 3
    losses = np.array([2.0, 2.01, 1.99, 2.02, 2.0, 1.98], np.float32)
    out = []
    for fused in (True, False):
        st = subzero.MatrixState(np.random.default_rng(5).standard_normal((m, n)) * 0.02, "f64", r)
        subzero.refresh(st, 4, 0, 0, reset_moments=True)
        subzero.run_step(st, 4, 0, 0, losses, "central", q, 1e-3, 1e-2, 0.9, 0.95, 1e-8, fused=fused)
        out.append(st.W)
    assert np.max(np.abs(out[0] - out[1])) < 1e-15


def _quadratic_losses(st, seed, i, t, q, eps, Wstar, scheme):
    """Exact losses L(W) = 1/2 ||W - W*||^2 at the points the plan visits."""
    passes, _ = subzero.pass_plan(scheme, q)
    W = st.W.copy()
    L = [] if scheme == "central" else [0.5 * np.sum((W - Wstar) ** 2)]
    for terms in passes:
        W = subzero.apply_pass(W, "f64", st.U, st.V,
                               subzero.perturb_coeff(seed, i, t, st.r, terms, eps))
        L.append(0.5 * np.sum((W - Wstar) ** 2))
    return np.array(L)


def test_central_estimator_on_a_quadratic_is_the_projected_directional_derivative():
    # For L(W) = 1/2 ||W - W*||^2 the central difference is exact:
    # rho_k = <grad L, U Z_k V^T> = <U^T (W - W*) V, Z_k>, so Eq. (6) gives
    # G = (1/q) sum_k <U^T grad V, Z_k> Z_k.
    m, n, r, q, eps = 20, 16, 4, 6, 1e-2
    rs = np.random.default_rng(7)
    st = subzero.MatrixState(rs.standard_normal((m, n)), "f64", r)
    subzero.refresh(st, 8, 0, 0, reset_moments=True)
    Wstar = rs.standard_normal((m, n))
    L = _quadratic_losses(st, 8, 0, 0, q, eps, Wstar, "central")
    rho = subzero.rho_from_losses(L, "central", eps, q)
    P = st.U.T @ (st.W - Wstar) @ st.V
    want = sum(np.sum(P * rng.gen_Z(8, 0, 0, k, r)) * rng.gen_Z(8, 0, 0, k, r) for k in range(q)) / q
    assert np.allclose(subzero.grad_G(8, 0, 0, r, rho), want, rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("scheme", ["central", "forward"])
def test_schedule_descends_a_quadratic(scheme):
    # A sign error anywhere (rho, G, the Adam direction, the -eta term, the
    # restore) makes this loss grow instead of fall.
    def run(lr):
        m, n, r, q, eps, T, F = 24, 20, 8, 8, 1e-3, 60, 10
        rs = np.random.default_rng(11)
        Wstar = rs.standard_normal((m, n)) * 0.1
        st = subzero.MatrixState(Wstar + rs.standard_normal((m, n)) * 0.1, "f64", r)
        L0 = 0.5 * np.sum((st.W - Wstar) ** 2)
        for t in range(T):
            if t % F == 0:
                subzero.refresh(st, 12, 0, t // F, reset_moments=(t == 0))
            L = _quadratic_losses(st, 12, 0, t, q, eps, Wstar, scheme)
            subzero.run_step(st, 12, 0, t, L, scheme, q, eps, lr, 0.9, 0.95, 1e-8)
        return 0.5 * np.sum((st.W - Wstar) ** 2) / L0

    assert run(2e-2) < 0.85
    assert run(-2e-2) > 1.2      # the same run with the update sign flipped ascends


def test_schedule_is_deterministic_and_restores_exactly_without_update():
    m, n, r, q = 16, 12, 4, 2
    W0 = rounding.round_to_bf16(np.random.default_rng(3).standard_normal((m, n)) * 0.02)
    loss_table = [np.full(2 * q, 2.0, np.float32)] * 4     # equal losses: rho = 0
    a = subzero.run_schedule(subzero.MatrixState(W0, "f64", r), 5, 1, loss_table, "central",
                             q, 4, 2, 1e-3, 1e-3, 0.9, 0.95, 1e-8)
    # rho = 0 -> G = 0 -> D = 0: the net change is zero in exact arithmetic
    assert np.max(np.abs(a.W - W0)) < 1e-15
    b1 = subzero.run_schedule(subzero.MatrixState(W0, "bf16", r), 5, 1, loss_table, "central",
                              q, 4, 2, 1e-1, 1e-3, 0.9, 0.95, 1e-8)
    b2 = subzero.run_schedule(subzero.MatrixState(W0, "bf16", r), 5, 1, loss_table, "central",
                              q, 4, 2, 1e-1, 1e-3, 0.9, 0.95, 1e-8)
    assert np.array_equal(b1.W, b2.W)

"""Mutation check of the oracle's pins (no GPU).

Each case plants one plausible mistake in the oracle, on the CPU and only for the length
of the case (a wrong Philox constant, a dropped Box-Muller factor, a skipped sign
correction, a transposed operand, a wrong Adam exponent, a wrong rounding mode, ...), then
runs the pins that guard that part of the oracle.  At least one pin must fail: a mistake
that every pin lets through would mean the oracle is not really pinned there.  The control
case runs the same pins on the unmutated oracle, so a failure under a mutant is the
mutant's doing.
"""

import math

import numpy as np
import pytest

import test_oracle_haar as P_haar
import test_oracle_linear as P_lin
import test_oracle_mezo as P_mezo
import test_oracle_rng as P_rng
import test_oracle_rounding as P_rnd
import test_oracle_subzero as P_sz
from conftest import read_golden_rows as golden
from oracle import haar, mezo, rng, rounding, subzero

# ---------------------------------------------------------------- the pins used here
PINS = {
    "philox_kat": lambda: P_rng.test_philox_known_answers(golden),
    "philox_layout": P_rng.test_philox_block_layout_matches_single_calls,
    "uniform": P_rng.test_uniform_exact_and_in_range,
    "box_muller": P_rng.test_box_muller_pairs_follow_the_definition,
    "normal_moments": P_rng.test_normals_moments_and_ks,
    "counter_fields": P_rng.test_counter_fields_select_independent_streams,
    "seed_key": lambda: P_rng.test_seed_splits_into_key_words((1 << 40) + 17),
    "bf16_library": P_rnd.test_bf16_matches_library_cast_on_fp32_inputs,
    "bf16_ties": P_rnd.test_bf16_ties_go_to_even,
    "bf16_half_ulp": P_rnd.test_bf16_is_idempotent_and_within_half_ulp,
    "qr_factorises": lambda: P_haar.test_householder_factorises(50, 10),
    "qr_lapack": lambda: P_haar.test_raw_factors_follow_lapack_convention(50, 10),
    "qr_unique": lambda: P_haar.test_sign_corrected_factor_is_the_unique_positive_diagonal_qr(50, 10),
    "sign_zero": P_haar.test_sign_correction_handles_zero_diagonal_as_plus_one,
    "haar_circle": P_haar.test_haar_m2_r1_angle_is_uniform_on_the_full_circle,
    "lemma1": lambda: P_sz.test_lemma1_isometry_and_projection(16, 12, 4),
    "restore": P_sz.test_perturb_then_restore_is_identity_in_exact_arithmetic,
    "round_once": P_sz.test_pass_rounds_once_to_storage_dtype,
    "rho": P_sz.test_rho_from_losses_schemes,
    "G": P_sz.test_G_single_query_unit_rho_is_Z_and_is_linear_in_rho,
    "adam_2x2": lambda: P_sz.test_adam_hand_computed_2x2(golden),
    "plans": lambda: P_sz.test_pass_plans_visit_the_paper_evaluation_points(4),
    "central_estimator": P_sz.test_central_estimator_on_a_quadratic_is_the_projected_directional_derivative,
    "descends_central": lambda: P_sz.test_schedule_descends_a_quadratic("central"),
    "descends_forward": lambda: P_sz.test_schedule_descends_a_quadratic("forward"),
    "no_update_restores": P_sz.test_schedule_is_deterministic_and_restores_exactly_without_update,
    "linear_hand": lambda: P_lin.test_hand_computed_1x2x2(golden),
    "linear_brute": lambda: P_lin.test_brute_force_definition(3, 5, 4, 2),
    "mezo_rows": P_mezo.test_row_streams_follow_the_counter_contract,
    "mezo_pass": P_mezo.test_perturb_restore_is_exact_in_fp64_and_rounds_once,
    "mezo_spsa": P_mezo.test_spsa_scalar_is_the_directional_derivative_of_a_quadratic,
}


def _fails(pin):
    try:
        with np.errstate(all="ignore"):
            PINS[pin]()
    except TypeError:          # a mutant called with the wrong arguments is a broken case,
        raise                  # not a caught mistake
    except Exception:          # an assertion, or an error the planted mistake provokes
        return True            # (a shape mismatch, say)
    return False


# ---------------------------------------------------------------- mistaken variants
def _philox(rounds=10, m0=rng.PHILOX_M0, m1=rng.PHILOX_M1, w0=rng.PHILOX_W0, w1=rng.PHILOX_W1,
            swap_outputs=False):
    """Philox4x32 with one of its parameters changed."""
    def f(ctr, key):
        msk = np.uint64(rng.MASK32)
        ctr = np.asarray(ctr, np.uint64) & msk
        key = np.asarray(key, np.uint64) & msk
        x0, x1, x2, x3 = ctr[..., 0], ctr[..., 1], ctr[..., 2], ctr[..., 3]
        k0, k1 = key[..., 0], key[..., 1]
        for rnd in range(rounds):
            if rnd > 0:
                k0, k1 = (k0 + np.uint64(w0)) & msk, (k1 + np.uint64(w1)) & msk
            p0, p1 = np.uint64(m0) * x0, np.uint64(m1) * x2
            hi0, lo0, hi1, lo1 = p0 >> np.uint64(32), p0 & msk, p1 >> np.uint64(32), p1 & msk
            if swap_outputs:
                x0, x1, x2, x3 = hi0 ^ x1 ^ k0, lo0, hi1 ^ x3 ^ k1, lo1
            else:
                x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
        return np.stack([x0, x1, x2, x3], axis=-1)
    return f


def _normals(kind):
    """Box-Muller with one mistake."""
    def f(seed, x1, x2, x3, n):
        n4 = (int(n) + 3) // 4 * 4
        u = rng.uniform_from_u32(rng.philox_block(seed, x1, x2, x3, n4).reshape(-1, 4))
        out = np.empty_like(u)
        for a, b in ((0, 1), (2, 3)):
            rad = np.sqrt((-1.0 if kind == "radius" else -2.0) * np.log(u[:, a]))
            ang = (1.0 if kind == "angle" else 2.0) * np.pi * u[:, b]
            c, s = np.cos(ang), np.sin(ang)
            out[:, a], out[:, b] = (s, c) if kind == "swap" else (c, s)
            out[:, a] *= rad
            out[:, b] *= rad
        return out.reshape(-1)[:n]
    return f


def _philox_block(kind):
    def f(seed, x1, x2, x3, n_words):
        n_ctr = (int(n_words) + 3) // 4
        c = np.arange(n_ctr, dtype=np.uint64)
        x3 = 0 if kind == "drop_query" else x3
        ctr = np.stack([c, np.full(n_ctr, int(x1) & rng.MASK32, np.uint64),
                        np.full(n_ctr, int(x2) & rng.MASK32, np.uint64),
                        np.full(n_ctr, int(x3) & rng.MASK32, np.uint64)], axis=-1)
        key = np.broadcast_to(np.array(rng.key_of_seed(seed), np.uint64), (n_ctr, 2))
        w = rng.philox4x32_10(ctr, key)
        if kind == "lane_major":
            w = w.T
        return w.reshape(-1)[:n_words]
    return f


def _round_bf16(kind):
    def f(x):
        x = np.asarray(x, np.float64)
        out = np.array(x, copy=True)
        fin = np.isfinite(x) & (x != 0.0)
        _, e = np.frexp(x[fin])
        q = np.ldexp(1.0, np.maximum(e - (7 if kind == "7bits" else 8), -133))
        y = x[fin] / q
        if kind == "half_away":
            y = np.sign(y) * np.floor(np.abs(y) + 0.5)
        elif kind == "truncate":
            y = np.trunc(y)
        else:
            y = np.rint(y)
        out[fin] = y * q
        return out
    return f


def _householder(kind):
    """Thin Householder QR (LAPACK reflector convention) with one mistake."""
    def f(A):
        A = np.array(A, np.float64, copy=True)
        m, r = A.shape
        taus = np.zeros(r)
        for j in range(r):
            x = A[j:, j]
            alpha, sigma = x[0], float(x[1:] @ x[1:])
            beta = -math.copysign(math.sqrt(alpha * alpha + sigma), alpha)
            tau = (beta - alpha) / (alpha if kind == "tau" else beta)
            v = x / (alpha - beta)
            v[0] = 1.0
            if j + 1 < r:
                A[j:, j + 1:] -= tau * np.outer(v, v @ A[j:, j + 1:])
            A[j, j] = beta
            A[j + 1:, j] = v[1:]
            taus[j] = tau
        R = np.triu(A[:r, :])
        Q = np.zeros((m, r))
        Q[:r, :r] = np.eye(r)
        order = range(r) if kind == "order" else reversed(range(r))
        for j in order:
            v = np.concatenate(([1.0], A[j + 1:, j]))
            Q[j:, :] -= taus[j] * np.outer(v, v @ Q[j:, :])
        return Q, R
    return f


def _gen_full_z(kind):
    def f(seed, i, t, n, rows):
        rows = np.asarray(rows, np.uint64)
        n4 = (n + 3) // 4
        stride = n // 4 if kind == "row_stride" else n4
        c = (rows[:, None] * np.uint64(stride) + np.arange(n4, dtype=np.uint64)[None, :]).reshape(-1)
        tag = rng.TAG_Z if kind == "tag" else mezo.TAG_MEZO
        ctr = np.stack([c, np.full(c.size, i, np.uint64), np.full(c.size, t, np.uint64),
                        np.full(c.size, rng.query_counter_word(tag, 0), np.uint64)], axis=-1)
        key = np.broadcast_to(np.array(rng.key_of_seed(seed), np.uint64), (c.size, 2))
        u = rng.uniform_from_u32(rng.philox4x32_10(ctr, key))
        z = np.empty_like(u)
        for a, b in ((0, 1), (2, 3)):
            rad = np.sqrt(-2.0 * np.log(u[:, a]))
            z[:, a], z[:, b] = rad * np.cos(2 * np.pi * u[:, b]), rad * np.sin(2 * np.pi * u[:, b])
        return z.reshape(rows.size, 4 * n4)[:, :n]
    return f


def _adam(kind):
    def f(M, Vm, G, beta1, beta2, eps_adam, adam_t):
        b1, b2 = float(beta1), float(beta2)
        if kind == "swap_betas":
            b1, b2 = b2, b1
        M_new = b1 * M + (1 - b1) * G
        Vm_new = b2 * Vm + (1 - b2) * (G if kind == "second_moment_G" else G * G)
        t = adam_t + 1 if kind == "exponent" else adam_t
        Mhat, Vhat = M_new / (1 - b1 ** t), Vm_new / (1 - b2 ** t)
        if kind == "eps_inside":
            D = Mhat / np.sqrt(Vhat + eps_adam)
        else:
            D = Mhat / (np.sqrt(Vhat) + eps_adam)
        return M_new, Vm_new, D, Mhat, Vhat
    return f


def _pass_plan(kind):
    good = subzero.pass_plan

    def f(scheme, q, fused=True):
        passes, restore = good(scheme, q, fused)
        if kind == "central_minus_one" and scheme == "central":
            passes = [[(k, -1.0) if c == -2.0 else (k, c) for k, c in terms] for terms in passes]
        if kind == "forward_restore_sign" and scheme == "forward":
            restore = [(k, -c) for k, c in restore]
        return passes, restore
    return f


def _rho(kind):
    good = subzero.rho_from_losses

    def f(losses, scheme, eps, q):
        rho = good(losses, scheme, eps, q)
        if kind == "central_sign" and scheme == "central":
            return -rho
        if kind == "forward_2eps" and scheme == "forward":
            return rho / 2.0
        return rho
    return f


MUTANTS = {
    # the counter-based generator (Philox4x32-10, uniform, Box-Muller, counter layout)
    "philox_multiplier": ([(rng, "philox4x32_10", _philox(m0=rng.PHILOX_M0 ^ 2))], ["philox_kat"]),
    "philox_9_rounds": ([(rng, "philox4x32_10", _philox(rounds=9))], ["philox_kat"]),
    "philox_weyl_increment": ([(rng, "philox4x32_10", _philox(w1=rng.PHILOX_W1 + 2))], ["philox_kat"]),
    "philox_output_order": ([(rng, "philox4x32_10", _philox(swap_outputs=True))], ["philox_kat"]),
    "key_words_swapped": ([(rng, "key_of_seed",
                            lambda s: ((int(s) >> 32) & rng.MASK32, int(s) & rng.MASK32))],
                          ["philox_layout", "seed_key"]),
    "uniform_without_offset": ([(rng, "uniform_from_u32",
                                 lambda x: (np.asarray(x, np.uint64) >> np.uint64(8)).astype(np.float64)
                                 * 2.0 ** -24)], ["uniform"]),
    "uniform_half_offset": ([(rng, "uniform_from_u32",
                              lambda x: ((np.asarray(x, np.uint64) >> np.uint64(8)).astype(np.float64)
                                         + 0.5) * 2.0 ** -24)], ["uniform"]),
    "box_muller_sin_cos_swapped": ([(rng, "normals", _normals("swap"))], ["box_muller"]),
    "box_muller_radius_factor": ([(rng, "normals", _normals("radius"))], ["box_muller", "normal_moments"]),
    "box_muller_half_angle": ([(rng, "normals", _normals("angle"))], ["box_muller", "normal_moments"]),
    "counter_drops_query": ([(rng, "philox_block", _philox_block("drop_query"))],
                            ["philox_layout", "counter_fields"]),
    "counter_lane_major": ([(rng, "philox_block", _philox_block("lane_major"))], ["philox_layout"]),
    # rounding to the storage dtype
    "bf16_ties_away_from_zero": ([(rounding, "round_to_bf16", _round_bf16("half_away"))],
                                 ["bf16_ties", "bf16_library"]),
    "bf16_seven_bits": ([(rounding, "round_to_bf16", _round_bf16("7bits"))], ["bf16_library"]),
    "bf16_truncation": ([(rounding, "round_to_bf16", _round_bf16("truncate"))],
                        ["bf16_library", "bf16_half_ulp"]),
    "pass_rounds_to_f32": ([(rounding, "round_to",
                             lambda x, dtype: rounding.round_to_f32(x) if dtype == "bf16"
                             else np.asarray(x, np.float64).copy())], ["round_once"]),
    # Alg. 1: Householder QR and the sign correction of Eq. (11)
    "sign_correction_skipped": ([(haar, "sign_correct", lambda Q, R: (Q, R))],
                                ["qr_unique", "haar_circle"]),
    "sign_from_Q_diagonal": ([(haar, "sign_correct",
                               lambda Q, R: (Q * np.where(np.diag(Q) < 0, -1.0, 1.0)[None, :],
                                             R * np.where(np.diag(Q) < 0, -1.0, 1.0)[:, None]))],
                             ["qr_unique"]),
    "sign_of_zero_is_zero": ([(haar, "sign_correct",
                               lambda Q, R: (Q * np.sign(np.diag(R))[None, :],
                                             R * np.sign(np.diag(R))[:, None]))], ["sign_zero"]),
    "householder_tau": ([(haar, "householder_qr", _householder("tau"))], ["qr_factorises", "qr_lapack"]),
    "householder_q_order": ([(haar, "householder_qr", _householder("order"))],
                            ["qr_factorises", "qr_lapack"]),
    # Eq. (4) / Lemma 1: the perturbation
    "delta_transposed_C": ([(subzero, "delta", lambda U, V, C: U @ (np.asarray(C).T @ V.T))],
                           ["lemma1"]),
    "delta_dropped_V": ([(subzero, "delta", lambda U, V, C: U @ C @ np.eye(C.shape[0], V.shape[0]))],
                        ["lemma1", "restore"]),
    "pass_ignores_row_subset": ([(subzero, "apply_pass",
                                  lambda W, dtype, U, V, C, rows=None:
                                  rounding.round_to(np.asarray(W) + subzero.delta(U, V, C), dtype))],
                                ["round_once"]),
    # Eqs. (3), (6): the scalars rho_k and the estimator
    "rho_central_sign": ([(subzero, "rho_from_losses", _rho("central_sign"))],
                         ["rho", "central_estimator", "descends_central"]),
    "rho_forward_over_2eps": ([(subzero, "rho_from_losses", _rho("forward_2eps"))], ["rho"]),
    "G_without_1_over_q": ([(subzero, "grad_G",
                             lambda seed, i, t, r, rho: sum(rho[k] * rng.gen_Z(seed, i, t, k, r)
                                                            for k in range(len(rho))))], ["G"]),
    "G_query_index_shifted": ([(subzero, "grad_G",
                                lambda seed, i, t, r, rho: sum(rho[k] * rng.gen_Z(seed, i, t, k + 1, r)
                                                               for k in range(len(rho))) / len(rho))],
                              ["G"]),
    # Eqs. (7)-(10): subspace Adam
    "adam_bias_exponent": ([(subzero, "adam", _adam("exponent"))], ["adam_2x2"]),
    "adam_eps_inside_sqrt": ([(subzero, "adam", _adam("eps_inside"))], ["adam_2x2"]),
    "adam_betas_swapped": ([(subzero, "adam", _adam("swap_betas"))], ["adam_2x2"]),
    "adam_second_moment_of_G": ([(subzero, "adam", _adam("second_moment_G"))], ["adam_2x2"]),
    # Eq. (10) fused with the restore, and the pass plans of Alg. 3
    "update_sign_flipped": ([(subzero, "step_coeff",
                              lambda D, lr, eps, terms, seed, i, t, r:
                              float(lr) * np.asarray(D) + sum(float(eps) * c * rng.gen_Z(seed, i, t, k, r)
                                                              for k, c in terms))],
                            ["descends_central", "descends_forward"]),
    "restore_dropped": ([(subzero, "step_coeff",
                          lambda D, lr, eps, terms, seed, i, t, r: -float(lr) * np.asarray(D))],
                        ["no_update_restores"]),
    "central_plan_minus_one": ([(subzero, "pass_plan", _pass_plan("central_minus_one"))],
                               ["plans", "no_update_restores"]),
    "forward_restore_sign": ([(subzero, "pass_plan", _pass_plan("forward_restore_sign"))],
                             ["plans", "descends_forward"]),
    # the perturbed linear layer
    "linear_drops_rank_r_term": ([(subzero, "perturbed_linear",
                                   lambda X, W, U, V, C, dtype="bf16":
                                   rounding.round_to(np.asarray(X) @ np.asarray(W).T, dtype))],
                                 ["linear_hand", "linear_brute"]),
    "linear_transposed_C": ([(subzero, "perturbed_linear",
                              lambda X, W, U, V, C, dtype="bf16":
                              rounding.round_to(np.asarray(X) @ (np.asarray(W)
                                                                 + U @ np.asarray(C).T @ V.T).T, dtype))],
                            ["linear_hand", "linear_brute"]),
    # MeZO's full-space perturbation (Eq. (1))
    "mezo_row_stride": ([(mezo, "gen_full_z", _gen_full_z("row_stride"))], ["mezo_rows"]),
    "mezo_tag": ([(mezo, "gen_full_z", _gen_full_z("tag"))], ["mezo_rows"]),
    "mezo_spsa_over_eps": ([(mezo, "spsa_rho", lambda lp, lm, eps: (float(lp) - float(lm)) / float(eps))],
                           ["mezo_spsa"]),
}


def test_pins_pass_on_the_unmutated_oracle():
    used = sorted({p for _, pins in MUTANTS.values() for p in pins})
    failing = [p for p in used if _fails(p)]
    assert not failing, failing


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_every_planted_mistake_fails_a_pin(name, monkeypatch):
    patches, pins = MUTANTS[name]
    for module, attr, value in patches:
        monkeypatch.setattr(module, attr, value)
    caught = [p for p in pins if _fails(p)]
    assert caught, f"mutant {name} passes every pin it should fail: {pins}"

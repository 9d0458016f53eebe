"""Full-space SPSA perturbation of MeZO (test infrastructure only).

Sec. 3, Eq. (1): the classical zeroth-order estimator perturbs every parameter,
w +- eps z with z ~ N(0, I_d), and MeZO regenerates z from a seed instead of
storing it.  Per matrix W (m x n) the in-place pass is

    W <- rnd(W + coef * Z),   Z[row, col] ~ N(0, 1) i.i.d.,

with coef = +eps, -2 eps, +eps (restore) for the two evaluations of Eq. (1), and
the SGD update W <- W - eta * rho * Z fused with the restore as coef = eps - eta rho.

Counter contract for Z (shared with the CUDA library by definition only):
Philox4x32-10 with key = seed, counter = (row * ceil(n / 4) + col // 4,
matrix index, t, 5 << 24), lane col % 4, then the uniform / Box-Muller
transform of ``oracle.rng``.  Each row starts on a fresh counter word, so a row's
normals do not depend on n mod 4.
"""

import numpy as np

from . import rng, rounding

TAG_MEZO = 5


def gen_full_z(seed, i, t, n, rows):
    """Rows `rows` (array of row indices) of Z (x n) for matrix i at step t, fp64."""
    rows = np.asarray(rows, dtype=np.uint64)
    n4 = (n + 3) // 4
    c = (rows[:, None] * np.uint64(n4) + np.arange(n4, dtype=np.uint64)[None, :]).reshape(-1)
    k = c.size
    ctr = np.stack([c,
                    np.full(k, int(i) & rng.MASK32, dtype=np.uint64),
                    np.full(k, int(t) & rng.MASK32, dtype=np.uint64),
                    np.full(k, rng.query_counter_word(TAG_MEZO, 0), dtype=np.uint64)], axis=-1)
    key = np.broadcast_to(np.array(rng.key_of_seed(seed), dtype=np.uint64), (k, 2))
    u = rng.uniform_from_u32(rng.philox4x32_10(ctr, key))
    z = np.empty_like(u)
    for a, b in ((0, 1), (2, 3)):
        rad = np.sqrt(-2.0 * np.log(u[:, a]))
        z[:, a] = rad * np.cos(2.0 * np.pi * u[:, b])
        z[:, b] = rad * np.sin(2.0 * np.pi * u[:, b])
    return z.reshape(rows.size, 4 * n4)[:, :n]


def mezo_pass(W, dtype, seed, i, t, coef, rows=None):
    """W <- rnd(W + coef * Z) (Eq. (1) perturbation, or the MeZO update), exact then
    rounded once.  With `rows`, W holds just those rows of the matrix."""
    W = np.asarray(W, np.float64)
    rows = np.arange(W.shape[0]) if rows is None else np.asarray(rows)
    Z = gen_full_z(seed, i, t, W.shape[1], rows)
    return rounding.round_to(W + float(coef) * Z, dtype)


def spsa_rho(loss_plus, loss_minus, eps):
    """Eq. (1)'s scalar: (L(w + eps z) - L(w - eps z)) / (2 eps)."""
    return (float(loss_plus) - float(loss_minus)) / (2.0 * float(eps))

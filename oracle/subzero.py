"""SubZero+ weight path of the oracle, one matrix at a time (test infrastructure only).

Plain fp64 restatement of Sec. 4 of the paper:

* ``perturbed_linear`` -- one linear layer of the loss evaluation of Alg. 3 at the
  perturbed weights, Y = X (W + U C V^T)^T, with W left as it is.
* ``perturb_coeff`` / ``apply_pass`` -- Alg. 2 (the in-place perturbation) and Eq. (4):
  W_i <- W_i + eps U_i Z_i V_i^T.  Consecutive updates that touch W with no
  loss evaluation in between (restore of query k, perturbation of query k+1,
  the Adam update) are summed into one r x r coefficient C and applied as ONE
  pass W <- rnd(W + U C V^T): exact in fp64, then rounded once to W's dtype.
* ``rho_from_losses`` -- Eq. (3) (central difference, pairs L+/L-) and the
  forward difference of Eq. (6) / Alg. 3 (rho_k = (l_k - l_0) / eps).
* ``grad_G``  -- Eq. (6) and the accumulation of Alg. 3:
  Zbar_i = (1/K) sum_k rho_k Z_i^(k) (K queries; called q in the code).
* ``adam``    -- Eqs. (7)-(10): moments, bias correction, the direction
  D = Mhat / (sqrt(Vhat) + eps_adam) that Eq. (10) applies as -eta U D V^T.
* ``run_schedule`` -- the Alg. 3 loop for one matrix: a refresh (Alg. 1) when
  t mod F == 0, the query passes, the Adam step fused with the final restore.

Readings of points the paper leaves open:
* the Adam exponent t in Eq. (9) is the count of Adam updates including the
  current one (``adam_t`` >= 1), since Alg. 3 starts at t = 0;
* moments are zeroed once (Alg. 3 first line) and kept across subspace
  refreshes unless ``reset_moments`` is set;
* V_i^t in Eq. (10) is the projection matrix, not the second moment; the
  second moment is called ``Vm`` here;
* eps_adam sits outside the square root (Eq. (10));
* every scalar hyper-parameter crosses the C boundary as fp32; callers pass
  the same fp32 values here.
"""

import numpy as np

from . import haar, rng, rounding

CENTRAL = "central"
FORWARD = "forward"
DIRECT = "direct"


# ----------------------------------------------------------------------------
# Alg. 2 / Eq. (4): one fused weight pass
# ----------------------------------------------------------------------------

def perturb_coeff(seed, i, t, r, terms, eps):
    """C = eps * sum_(k, c) c * Z_i^(k) at step t, for terms [(k, c), ...]."""
    C = np.zeros((r, r))
    for k, c in terms:
        C += float(c) * rng.gen_Z(seed, i, t, k, r)
    return float(eps) * C


def delta(U, V, C):
    """Exact fp64 U C V^T (Lemma 1 form of Eq. (4))."""
    return np.asarray(U, np.float64) @ (np.asarray(C, np.float64) @ np.asarray(V, np.float64).T)


def apply_pass(W, dtype, U, V, C, rows=None):
    """W <- rnd_dtype(W + U C V^T).  ``rows`` restricts the pass to a row subset
    (the rows of W given), which is exact because each row is independent."""
    W = np.asarray(W, np.float64)
    Uu = np.asarray(U, np.float64) if rows is None else np.asarray(U, np.float64)[rows]
    return rounding.round_to(W + delta(Uu, V, C), dtype)


def perturbed_linear(X, W, U, V, C, dtype="bf16"):
    """Y = X (W + U C V^T)^T: a linear layer y = W' x (nn.Linear's W, out x in) applied to
    the rows of X at the perturbed weights W' = W + U C V^T at which Alg. 3 evaluates the
    loss, without W' being written anywhere.  Exact in fp64, rounded once to ``dtype``.
    (The weight-pass form evaluates the same layer at rnd(W + U C V^T), a weight already
    rounded to W's storage type.)"""
    X = np.asarray(X, np.float64)
    Wp = np.asarray(W, np.float64) + delta(U, V, C)
    return rounding.round_to(X @ Wp.T, dtype)


# ----------------------------------------------------------------------------
# Eq. (3) / Eq. (6): the scalars rho_k and the in-subspace gradient
# ----------------------------------------------------------------------------

def rho_from_losses(losses, scheme, eps, q):
    """rho_k, k = 0..q-1, in fp64 from the fp32 losses.

    central: losses = [L+_0, L-_0, L+_1, L-_1, ...] (2q), rho_k = (L+_k - L-_k)/(2 eps)  (Eq. (3))
    forward: losses = [l_0, l_1, ..., l_q] (q+1),       rho_k = (l_(k+1) - l_0)/eps     (Eq. (6), Alg. 3)
    direct : losses = [rho_0, ..., rho_(q-1)] (q)
    """
    L = np.asarray(losses, dtype=np.float64)
    eps = float(eps)
    if scheme == CENTRAL:
        assert L.size == 2 * q
        return (L[0::2] - L[1::2]) / (2.0 * eps)
    if scheme == FORWARD:
        assert L.size == q + 1
        return (L[1:] - L[0]) / eps
    if scheme == DIRECT:
        assert L.size == q
        return L.copy()
    raise ValueError(scheme)


def grad_G(seed, i, t, r, rho):
    """Zbar_i = (1/q) sum_k rho_k Z_i^(k): accumulate in k order, then divide (Alg. 3)."""
    q = len(rho)
    G = np.zeros((r, r))
    for k in range(q):
        G += rho[k] * rng.gen_Z(seed, i, t, k, r)
    return G / q


# ----------------------------------------------------------------------------
# Eqs. (7)-(10): subspace Adam
# ----------------------------------------------------------------------------

def adam(M, Vm, G, beta1, beta2, eps_adam, adam_t):
    """One subspace-Adam update of the r x r moments.

    Returns (M_new, Vm_new, D, Mhat, Vhat) with D = Mhat / (sqrt(Vhat) + eps_adam),
    the matrix that Eq. (10) applies as W <- W - eta U D V^T.
    """
    b1, b2 = float(beta1), float(beta2)
    M_new = b1 * np.asarray(M, np.float64) + (1.0 - b1) * G                 # Eq. (7)
    Vm_new = b2 * np.asarray(Vm, np.float64) + (1.0 - b2) * (G * G)         # Eq. (8)
    Mhat = M_new / (1.0 - b1 ** int(adam_t))                                # Eq. (9)
    Vhat = Vm_new / (1.0 - b2 ** int(adam_t))
    D = Mhat / (np.sqrt(Vhat) + float(eps_adam))                            # Eq. (10)
    return M_new, Vm_new, D, Mhat, Vhat


def sgd_direction(G):
    """SubZero's plain SGD in the subspace (Sec. 3): the update direction is G itself."""
    return np.asarray(G, np.float64).copy()


def step_coeff(D, lr, eps, restore_terms, seed, i, t, r):
    """C = -lr D + eps * sum_(k, c) c Z_i^(k): the Adam update of Eq. (10) fused
    with the restore of the last query (Alg. 3, its second perturbation call)."""
    C = -float(lr) * np.asarray(D, np.float64)
    for k, c in restore_terms:
        C = C + float(eps) * float(c) * rng.gen_Z(seed, i, t, k, r)
    return C


# ----------------------------------------------------------------------------
# Alg. 3: the per-step pass plan and the schedule driver
# ----------------------------------------------------------------------------

def pass_plan(scheme, q, fused=True):
    """Weight passes of one step: (perturb_passes, restore_terms).

    perturb_passes: list of term lists [(k, c), ...]; each is one rounded pass
    W += eps U (sum c Z_k) V^T followed by one loss evaluation.
    restore_terms: the terms fused into the final Adam pass.

    central (Eq. (3), loss pairs): +Z0 | -2Z0 | +Z0+Z1 | -2Z1 | ... | -2Z_(q-1); restore +Z_(q-1)
    forward (Alg. 3):              +Z0 | Z1-Z0 | ... | Z_(q-1)-Z_(q-2);         restore -Z_(q-1)
    With fused=False every perturbation call of Alg. 3 is its own rounded pass
    (restores become separate passes with no loss evaluation after them).
    """
    passes = []
    if scheme == CENTRAL:
        if fused:
            for k in range(q):
                passes.append([(k, 1.0)] if k == 0 else [(k - 1, 1.0), (k, 1.0)])
                passes.append([(k, -2.0)])
            return passes, [(q - 1, 1.0)]
        for k in range(q):
            passes += [[(k, 1.0)], [(k, -2.0)], [(k, 1.0)]]
        return passes, []
    if scheme == FORWARD:
        if fused:
            for k in range(q):
                passes.append([(k, 1.0)] if k == 0 else [(k, 1.0), (k - 1, -1.0)])
            return passes, [(q - 1, -1.0)]
        for k in range(q):
            passes += [[(k, 1.0)], [(k, -1.0)]]
        return passes, []
    raise ValueError(scheme)


class MatrixState:
    """State of one trainable matrix W_i (m x n) and its r x r optimizer buffers."""

    def __init__(self, W, dtype, r):
        self.W = np.asarray(W, np.float64).copy()
        self.dtype = dtype
        self.m, self.n = self.W.shape
        self.r = r
        self.U = None
        self.V = None
        self.M = np.zeros((r, r))
        self.Vm = np.zeros((r, r))
        self.adam_t = 0


def refresh(state, seed, i, j, reset_moments=False):
    """Alg. 3's refresh: new bases U, V from Alg. 1 every F steps."""
    state.U, state.V = haar.haar_proj(seed, i, j, state.m, state.n, state.r)
    if reset_moments:
        state.M[:] = 0.0
        state.Vm[:] = 0.0
        state.adam_t = 0


def run_step(state, seed, i, t, losses, scheme, q, eps, lr, beta1, beta2, eps_adam,
             fused=True, optimizer="adam"):
    """One Alg. 3 iteration for one matrix (given the step's losses). Returns G."""
    passes, restore = pass_plan(scheme, q, fused)
    for terms in passes:
        C = perturb_coeff(seed, i, t, state.r, terms, eps)
        state.W = apply_pass(state.W, state.dtype, state.U, state.V, C)
    rho = rho_from_losses(losses, scheme, eps, q)
    G = grad_G(seed, i, t, state.r, rho)
    if optimizer == "adam":
        state.adam_t += 1
        state.M, state.Vm, D, _, _ = adam(state.M, state.Vm, G, beta1, beta2, eps_adam,
                                          state.adam_t)
    else:
        D = sgd_direction(G)
    C = step_coeff(D, lr, eps, restore, seed, i, t, state.r)
    state.W = apply_pass(state.W, state.dtype, state.U, state.V, C)
    return G


def run_schedule(state, seed, i, loss_table, scheme, q, T, F, eps, lr, beta1, beta2,
                 eps_adam, reset_moments=False, fused=True, t0=0, optimizer="adam"):
    """Alg. 3 for one matrix over steps t0..T-1 (refresh j = t // F when t mod F == 0)."""
    for t in range(t0, T):
        if t % F == 0:
            refresh(state, seed, i, t // F, reset_moments=(reset_moments or t == 0))
        run_step(state, seed, i, t, loss_table[t], scheme, q, eps, lr, beta1, beta2,
                 eps_adam, fused=fused, optimizer=optimizer)
    return state

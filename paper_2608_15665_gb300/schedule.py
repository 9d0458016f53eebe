"""Caller-side helpers around the C ABI: buffers per matrix and the Alg. 3 call order.

``SubZeroPlus`` allocates U, V (fp32 bases) and M, Vm (fp32 moments) next to each
caller-owned weight tensor and binds them into one context.  ``step_plan`` lists
the zo_perturb calls of one step -- the places where the caller evaluates a
loss -- and the restore term handed to zo_step:

* central scheme (Eq. (3), loss pairs): evaluate at W + eps Z_k and W - eps Z_k:
    +Z_0 | -2 Z_0 | +Z_0 +Z_1 | -2 Z_1 | ... | -2 Z_(q-1)   then restore +Z_(q-1)
* forward scheme (Alg. 3, Eq. (6)): evaluate at W + eps Z_k (after one at W):
    +Z_0 | +Z_1 -Z_0 | ... | +Z_(q-1) -Z_(q-2)              then restore -Z_(q-1)
Each entry is ((qa, ca), (qb, cb) or None).  ``linear_plan`` lists the same evaluation
points for the route that never writes the perturbation into W (zo_linear_prepare /
zo_linear_perturbed feed W + eps U Z V^T straight into the forward GEMMs): there each entry
is the absolute perturbation of one loss evaluation, and zo_step then has nothing to
restore.  No arithmetic happens here.
"""

import torch

from . import binding as zb

SCHEMES = {"central": zb.ZO_SCHEME_CENTRAL, "forward": zb.ZO_SCHEME_FORWARD,
           "direct": zb.ZO_SCHEME_DIRECT}


def step_plan(scheme, q):
    if scheme == "central":
        calls = []
        for k in range(q):
            calls.append(((k, 1.0), None) if k == 0 else ((k - 1, 1.0), (k, 1.0)))
            calls.append(((k, -2.0), None))
        return calls, (q - 1, 1.0)
    if scheme == "forward":
        calls = [((0, 1.0), None)] + [((k, 1.0), (k - 1, -1.0)) for k in range(1, q)]
        return calls, (q - 1, -1.0)
    raise ValueError(f"no pass plan for scheme {scheme!r}")


def linear_plan(scheme, q):
    """The loss evaluations of one step on the perturbed-linear route: ((qa, ca), None) for
    the evaluation at W + eps ca Z_qa (ca = 0: at W itself)."""
    if scheme == "central":
        return [((k, c), None) for k in range(q) for c in (1.0, -1.0)]
    if scheme == "forward":
        return [((0, 0.0), None)] + [((k, 1.0), None) for k in range(q)]
    raise ValueError(f"no evaluation plan for scheme {scheme!r}")


class SubZeroPlus:
    """One context over a list of weight tensors (bf16 or fp32, on one CUDA device)."""

    def __init__(self, weights, r, q, seed, matrix_index_base=0, stream=None):
        self.weights = list(weights)
        self.r, self.q, self.seed = int(r), int(q), int(seed)
        dev = self.weights[0].device
        f32 = dict(dtype=torch.float32, device=dev)
        self.U = [torch.empty(W.shape[0], r, **f32) for W in self.weights]
        self.V = [torch.empty(W.shape[1], r, **f32) for W in self.weights]
        self.M = [torch.zeros(r, r, **f32) for _ in self.weights]
        self.Vm = [torch.zeros(r, r, **f32) for _ in self.weights]
        mats = [zb.make_matrix(W, U, V, M, Vm)
                for W, U, V, M, Vm in zip(self.weights, self.U, self.V, self.M, self.Vm)]
        self.stream = stream
        self.ctx = zb.zo_create(mats, r, q, seed, matrix_index_base, stream)

    # -- thin forwards of the C ABI ---------------------------------------------
    def init_subspace(self, refresh_idx=0):
        zb.zo_init_subspace(self.ctx, refresh_idx)

    def refresh(self, refresh_idx, reset_moments=False):
        zb.zo_refresh(self.ctx, refresh_idx, reset_moments)

    def perturb(self, t, qa, ca, qb=-1, cb=0.0, eps=1e-3):
        zb.zo_perturb(self.ctx, t, qa, ca, qb, cb, eps)

    def step(self, t, adam_t, losses, scheme, eps, lr, beta1, beta2, eps_adam, restore_query,
             restore_coef, optimizer=zb.ZO_OPT_ADAM, gamma_out=None):
        zb.zo_step(self.ctx, t, adam_t, losses, SCHEMES[scheme], eps, lr, beta1, beta2, eps_adam,
                   restore_query, restore_coef, optimizer, gamma_out)

    def linear_prepare(self, t, qa, ca, qb=-1, cb=0.0, eps=1e-3):
        """Prepare the linear layers' evaluation at W + eps (ca Z_qa + cb Z_qb) (every W
        left as it is)."""
        zb.zo_linear_prepare(self.ctx, t, qa, ca, qb, cb, eps)

    def linear_perturbed(self, i, X, Y=None):
        """Y = X (W_i + U_i C V_i^T)^T for the prepared C (bf16 X of T x n_i; Y allocated
        as T x m_i bf16 if not given)."""
        if Y is None:
            Y = torch.empty(X.shape[0], self.weights[i].shape[0], dtype=torch.bfloat16,
                            device=X.device)
        zb.zo_linear_perturbed(self.ctx, i, X, Y)
        return Y

    def mezo_perturb(self, t, coef):
        """Full-space SPSA pass of Eq. (1): every W_i <- rnd(W_i + coef Z_i)."""
        zb.zo_mezo_perturb(self.ctx, t, coef)

    def sync(self):
        zb.zo_sync_status(self.ctx)

    def close(self):
        if self.ctx is not None:
            zb.zo_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- one step of Alg. 3 ----------------------------------------------------
    def run_step(self, t, adam_t, loss_fn, scheme, eps, lr, beta1, beta2, eps_adam,
                 optimizer=zb.ZO_OPT_ADAM, gamma_out=None):
        """Alg. 3 for one step: the perturbation passes with a loss evaluation after
        each (``loss_fn(t, index)`` returns the caller's loss; for the forward scheme
        it is called once more first, at the unperturbed weights), then zo_step."""
        calls, (rq, rc) = step_plan(scheme, self.q)
        losses = [loss_fn(t, 0)] if scheme == "forward" else []
        for (qa, ca), second in calls:
            qb, cb = second if second is not None else (-1, 0.0)
            self.perturb(t, qa, ca, qb, cb, eps)
            losses.append(loss_fn(t, len(losses)))
        self.step(t, adam_t, losses, scheme, eps, lr, beta1, beta2, eps_adam, rq, rc, optimizer,
                  gamma_out)
        return losses

    def run_step_linear(self, t, adam_t, loss_fn, scheme, eps, lr, beta1, beta2, eps_adam,
                        optimizer=zb.ZO_OPT_ADAM, gamma_out=None):
        """Alg. 3 for one step with every loss evaluated at the perturbed weights inside the
        forward GEMMs: before each ``loss_fn(t, index)`` (whose forward calls
        ``linear_perturbed``) the evaluation point is prepared; W is written once, by
        zo_step's update (nothing to restore)."""
        losses = []
        for (qa, ca), _ in linear_plan(scheme, self.q):
            self.linear_prepare(t, qa, ca, -1, 0.0, eps)
            losses.append(loss_fn(t, len(losses)))
        self.step(t, adam_t, losses, scheme, eps, lr, beta1, beta2, eps_adam, -1, 0.0, optimizer,
                  gamma_out)
        return losses

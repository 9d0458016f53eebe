"""GPU parity of the full-space SPSA perturbation of Eq. (1) (zo_mezo_perturb)."""

import numpy as np
import pytest
import torch

from gpu_util import f32, make_weight, snapshot
from oracle import mezo
from parity import NORMAL_ABS, assert_weights

pytestmark = pytest.mark.gpu

# bf16 and fp32, ragged rows/columns (n not a multiple of 4 or 8), a padded row stride
SHAPES = [(300, 520, "bf16", None), (33, 1000, "bf16", 1008), (70, 36, "bf16", 40),
          (129, 130, "f32", 132), (8, 5120, "f32", None)]


def _ctx(gpu, seed, base):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    weights = [make_weight(m, n, dt, 50 + k, gpu, ldw) for k, (m, n, dt, ldw) in enumerate(SHAPES)]
    return SubZeroPlus(weights, 4, 2, seed, matrix_index_base=base)


@pytest.mark.parametrize("coef", [1e-3, -2e-3, 0.25])
def test_mezo_pass_matches_oracle(lib, gpu, coef):
    seed, base, t = 31337, 7, 12
    z = _ctx(gpu, seed, base)
    before = snapshot(z)
    z.mezo_perturb(t, coef)
    after = snapshot(z)
    c = f32(coef)
    for i, (m, n, dt, _) in enumerate(SHAPES):
        want = mezo.mezo_pass(before["W"][i], dt, seed, base + i, t, c)
        T = np.abs(c * mezo.gen_full_z(seed, base + i, t, n, np.arange(m)))
        assert_weights(after["W"][i], want, dt, f"mezo matrix {i}", before=before["W"][i],
                       terms=(T, abs(c) * NORMAL_ABS))
    z.sync()
    z.close()


def test_mezo_spsa_cycle_restores_and_updates(lib, gpu):
    # +eps, -2 eps, then restore fused with the SGD update: eps - lr * rho
    seed, base, t, eps, lr = 99, 0, 3, 1e-3, 1e-4
    z = _ctx(gpu, seed, base)
    W0 = snapshot(z)["W"]
    rho = mezo.spsa_rho(2.01, 1.99, f32(eps))
    for coef in (eps, -2 * eps, eps - lr * rho):
        z.mezo_perturb(t, coef)
    got = snapshot(z)["W"]
    for i, (m, n, dt, _) in enumerate(SHAPES):
        W = W0[i]
        for coef in (eps, -2 * eps, eps - lr * rho):
            W = mezo.mezo_pass(W, dt, seed, base + i, t, f32(coef))
        # three rounded passes: compare normwise against the oracle's trajectory
        scale = np.abs(W0[i]).max()
        if dt == "bf16":
            assert np.max(np.abs(got[i] - W)) <= 4 * 2.0 ** -8 * scale
        else:
            assert np.max(np.abs(got[i] - W)) <= 1e-5 * scale
        # the net change is -lr * rho * Z up to rounding
        Z = mezo.gen_full_z(seed, base + i, t, n, np.arange(m))
        if dt == "f32":
            assert np.allclose(got[i] - W0[i], -lr * rho * Z, atol=1e-6 * scale)
    z.close()

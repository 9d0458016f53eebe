"""GPU parity of the full-space SPSA perturbation of Eq. (1) (zo_mezo_perturb)."""

import numpy as np
import pytest
import torch

from gpu_util import f32, make_weight, snapshot
from oracle import mezo, rounding
from parity import NORMAL_ABS, assert_normwise, assert_weights

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
    # +eps, -2 eps, then restore fused with the SGD update: eps - lr * rho.  Every pass is
    # checked element by element against the oracle's pass on the same input; the three-pass
    # result against the oracle's own three-pass trajectory, where an element may differ only
    # if one of its passes had the exact value within the pass's evaluation error of a bf16
    # rounding boundary (fp32 Gaussians within NORMAL_ABS, one fp32 fma, then the rounding).
    from parity import U24, bf16_boundary_distance
    seed, base, t, eps, lr = 99, 0, 3, 1e-3, 1e-4
    z = _ctx(gpu, seed, base)
    W0 = snapshot(z)["W"]
    rho = mezo.spsa_rho(2.01, 1.99, f32(eps))
    coefs = (eps, -2 * eps, eps - lr * rho)
    for coef in coefs:
        before = snapshot(z)["W"]
        z.mezo_perturb(t, coef)
        after = snapshot(z)["W"]
        c = f32(coef)
        for i, (m, n, dt, _) in enumerate(SHAPES):
            want = mezo.mezo_pass(before[i], dt, seed, base + i, t, c)
            T = np.abs(c * mezo.gen_full_z(seed, base + i, t, n, np.arange(m)))
            assert_weights(after[i], want, dt, f"mezo cycle pass {coef:.3e}, matrix {i}",
                           before=before[i], terms=(T, abs(c) * NORMAL_ABS))
    got = snapshot(z)["W"]
    for i, (m, n, dt, _) in enumerate(SHAPES):
        Z = mezo.gen_full_z(seed, base + i, t, n, np.arange(m))
        W, near = W0[i], np.zeros(W0[i].shape, np.int64)
        for coef in coefs:
            c = f32(coef)
            x = W + c * Z
            if dt == "bf16":
                near += bf16_boundary_distance(x) <= abs(c) * (NORMAL_ABS + U24 * np.abs(Z)) + U24 * np.abs(x)
            W = mezo.mezo_pass(W, dt, seed, base + i, t, c)
        if dt == "bf16":
            differ = got[i] != W
            assert not (differ & (near == 0)).any(), f"matrix {i}: differs away from a rounding boundary"
            # at most 2 ulps per near-boundary pass, ulps at max(|W|, rms W0) (weights near zero)
            rms = float(np.sqrt(np.mean(W0[i] ** 2)))
            ulp = rounding.bf16_ulp(np.maximum.reduce([np.abs(W), np.abs(got[i]), np.full(W.shape, rms)]))
            assert np.all(np.abs(got[i] - W) <= 2 * near * ulp)
        else:
            assert_normwise(got[i], W, f"mezo cycle, matrix {i}")
            # the net change is -lr * rho * Z up to rounding
            assert np.allclose(got[i] - W0[i], -lr * rho * Z, atol=1e-6 * np.abs(W0[i]).max())
    z.close()

"""GPU parity of the refresh (Alg. 1 / Eq. (11)): CholeskyQR2 for panels with >= 4r rows at
r >= 16, batched TSQR + sign correction for the others -- both must give the unique
positive-diagonal factor of the oracle."""

import numpy as np
import pytest
import torch

from gpu_util import make_weight, snapshot
from oracle import haar, rng
from parity import UV_ABS

pytestmark = pytest.mark.gpu

CASES = [
    (4, [(8, 5120), (5120, 8), (4097, 9)]),          # LoRA shapes; two level-0 blocks + ragged
    (8, [(256, 256), (2049, 300)]),
    (16, [(2048, 8192), (1500, 40)]),
    (32, [(11008, 4096), (600, 33)]),                # three-level tree for 11008 rows
    (64, [(25600, 128), (300, 64), (64, 257)]),      # five levels for 25600 rows; m == r
    (128, [(2048, 130), (300, 256)]),                 # four levels for 2048 rows; ragged tail
    (16, [(64, 63), (1025, 64)]),                    # rows = 4r (CholeskyQR2) next to 4r - 1 (TSQR)
    (32, [(128, 127), (2049, 128)]),                 # the same at r = 32; a 1-row last chunk
]


@pytest.mark.parametrize("r,shapes", CASES, ids=[f"r{c[0]}-{k}" for k, c in enumerate(CASES)])
def test_refresh_matches_oracle(lib, gpu, r, shapes):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    seed, base = 4242 + r, 10
    # W rows must start on 16-byte boundaries: pad the row stride, keep n ragged
    weights = [make_weight(m, n, "bf16", k, gpu, ldw=(n + 7) // 8 * 8) for k, (m, n) in enumerate(shapes)]
    z = SubZeroPlus(weights, r, 2, seed, matrix_index_base=base)
    for j in (0, 3):
        z.refresh(j, reset_moments=True)
        s = snapshot(z)
        for i, (m, n) in enumerate(shapes):
            U, V = haar.haar_proj(seed, base + i, j, m, n, r)
            for got, want, om_which, rows in ((s["U"][i], U, "U", m), (s["V"][i], V, "V", n)):
                assert np.max(np.abs(got - want)) <= UV_ABS, (i, om_which)
                assert np.max(np.abs(got.T @ got - np.eye(r))) <= 1e-5
                # Q^T Omega is R: upper triangular with a positive diagonal (Eq. (11))
                om = rng.gen_omega(seed, base + i, j, om_which, rows, r)
                R = got.T @ om
                assert np.all(np.diag(R) > 0)
                assert np.max(np.abs(np.tril(R, -1))) <= 1e-4 * np.abs(np.diag(R)).max()
    z.close()


def test_refresh_resets_moments_only_when_asked(lib, gpu):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    z = SubZeroPlus([make_weight(64, 64, "f32", 1, gpu)], 8, 2, 5)
    z.init_subspace(0)
    z.M[0].fill_(1.5)
    z.Vm[0].fill_(2.5)
    z.refresh(1, reset_moments=False)
    torch.cuda.synchronize()
    assert float(z.M[0].min()) == 1.5 and float(z.Vm[0].max()) == 2.5
    z.refresh(2, reset_moments=True)
    torch.cuda.synchronize()
    assert float(z.M[0].abs().max()) == 0.0 and float(z.Vm[0].abs().max()) == 0.0
    z.close()


def test_refresh_is_deterministic(lib, gpu):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    z = SubZeroPlus([make_weight(3000, 704, "bf16", 2, gpu)], 32, 2, 77)
    z.refresh(5)
    a = [z.U[0].clone(), z.V[0].clone()]
    z.refresh(6)
    z.refresh(5)
    torch.cuda.synchronize()
    assert torch.equal(a[0], z.U[0]) and torch.equal(a[1], z.V[0])
    z.close()

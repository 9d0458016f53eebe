"""The layer partition on the GPU, in one process: a set split over two contexts (matrix
indices 0 .. n-1 and n .. 2n-1 through matrix_index_base) must give, bit for bit, what one
context over the whole set gives.  Every matrix's update depends only on its own state, the
shared seed, its global index and the shared losses (Alg. 3), so this is the property the
multi-GPU layer partition rests on; each rank of bench.py is one such context."""

import numpy as np
import pytest
import torch

from gpu_util import make_weight

pytestmark = pytest.mark.gpu

# (dtype, r, shapes): the FMA pass, the tensor-core pass with both operands in shared memory,
# and the one with U in Tensor Memory
CASES = [("f32", 8, [(300, 520), (130, 1000), (96, 64), (520, 300)]),
         ("bf16", 32, [(300, 520), (1030, 264), (512, 384), (264, 136)]),
         ("bf16", 64, [(512, 264), (1030, 136), (264, 512), (640, 256)])]


def _run(z, table, steps, F, eps=1e-2):
    for t in range(steps):
        if t % F == 0:
            z.refresh(t // F, reset_moments=(t == 0))
        z.run_step(t, t + 1, lambda tt, k: float(table[tt][k]), "central", eps, 1e-2, 0.9, 0.95, 1e-8)


@pytest.mark.parametrize("dtype,r,shapes", CASES, ids=[f"{c[0]}-r{c[1]}" for c in CASES])
def test_two_contexts_over_halves_equal_one_over_the_whole_set(lib, gpu, dtype, r, shapes):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    seed, q, steps, F = 4242, 4, 4, 3
    table = (2.0 + 0.01 * np.random.default_rng(11).standard_normal((steps, 2 * q))).astype(np.float32)
    W0 = [make_weight(m, n, dtype, 30 + k, gpu) for k, (m, n) in enumerate(shapes)]
    half = len(shapes) // 2
    whole = SubZeroPlus([W.clone() for W in W0], r, q, seed)
    parts = [SubZeroPlus([W.clone() for W in W0[:half]], r, q, seed, matrix_index_base=0),
             SubZeroPlus([W.clone() for W in W0[half:]], r, q, seed, matrix_index_base=half)]
    for z in [whole] + parts:
        _run(z, table, steps, F)
    want_path = 1 if dtype == "f32" else 2
    assert zb.zo_wpass_path(whole.ctx) == want_path
    torch.cuda.synchronize()
    for k in range(len(shapes)):
        z, j = (parts[0], k) if k < half else (parts[1], k - half)
        for name in ("weights", "U", "V", "M", "Vm"):
            a, b = getattr(z, name)[j], getattr(whole, name)[k]
            assert torch.equal(a, b), f"matrix {k}: {name} differs between the split and the whole set"
    assert not torch.equal(whole.weights[0], W0[0])           # the steps did move W
    for z in [whole] + parts:
        z.sync()
        z.close()

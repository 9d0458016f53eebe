"""GPU test of zo_perturb_noalloc, the entry point for callers that cannot allocate
device memory (their GPU memory belongs to another allocator's pool, or they cannot
afford the synchronisation cudaMalloc may cause).  It must compute what the
context-based zo_perturb computes, using only its built-in 8 MiB scratch array.

Kept in a file of its own that pytest collects last."""

import numpy as np
import pytest
import torch

from gpu_util import make_weight
from parity import assert_weights, to_f64

pytestmark = pytest.mark.gpu

CASES = [("f32", 8, 300, 520), ("bf16", 32, 1030, 264), ("bf16", 64, 200, 5120)]


@pytest.mark.parametrize("dtype,r,m,n", CASES)
def test_noalloc_matches_zo_perturb_on_two_calls(lib, gpu, dtype, r, m, n):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    seed, base, eps = 8080, 17, 1e-1
    W0 = make_weight(m, n, dtype, 5, gpu)
    z = SubZeroPlus([W0.clone()], r, 4, seed, matrix_index_base=base)
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, 1)   # the fp32-FMA arithmetic of the variant
    z.init_subspace(0)
    W = W0.clone()
    for t, qa, ca, qb, cb in [(0, 0, 1.0, -1, 0.0), (0, 0, -2.0, 1, 1.0)]:
        before = to_f64(z.weights[0])
        z.perturb(t, qa, ca, qb, cb, eps)
        zb.zo_perturb_noalloc(W, z.U[0], z.V[0], r, seed, base, t, qa, ca, qb, cb, eps)
        torch.cuda.synchronize()
        assert_weights(to_f64(W), to_f64(z.weights[0]), dtype, f"no-alloc t={t} qa={qa}",
                       before=before)
    assert not torch.equal(W, W0)                         # the passes did change W
    z.sync()
    z.close()


def test_noalloc_rejects_requests_beyond_its_scratch(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    W = torch.zeros(64, 40000, dtype=torch.float32, device=gpu)
    U = torch.zeros(64, 64, dtype=torch.float32, device=gpu)
    V = torch.zeros(40000, 64, dtype=torch.float32, device=gpu)
    with pytest.raises(zb.ZoError) as e:
        zb.zo_perturb_noalloc(W, U, V, 64, 1, 0, 0, 0, 1.0, -1, 0.0, 1e-3)
    assert e.value.status == zb.ZO_ERR_SHAPE and "8 MiB" in str(e.value)
    torch.cuda.synchronize()
    assert float(W.abs().max()) == 0.0

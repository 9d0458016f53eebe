"""GPU test of zo_perturb_noalloc, the entry point for callers that cannot allocate
device memory: code whose GPU memory belongs to another allocator's pool (a framework's
caching allocator that has reserved the device, where a stray cudaMalloc fails or
fragments it), or loops that cannot afford the device synchronisation cudaMalloc and
cudaFree may cause.  It must compute exactly what the context-based zo_perturb computes
on its FMA path -- the same kernels, with their scratch in the library's built-in 8 MiB
array -- and match the oracle; and it must leave the device's free memory unchanged.

Kept in a file of its own that pytest collects last."""

import numpy as np
import pytest
import torch

from gpu_util import f32, make_weight
from oracle import subzero
from parity import assert_weights, to_f64, update_terms

pytestmark = pytest.mark.gpu

# (dtype, r, m, n): the last is wider than 256 projection units of 128 columns
CASES = [("f32", 8, 300, 520), ("bf16", 32, 1030, 264), ("bf16", 64, 200, 5120),
         ("bf16", 8, 40, 40000), ("f32", 4, 24, 33000)]


@pytest.mark.parametrize("dtype,r,m,n", CASES, ids=[f"{c[0]}-r{c[1]}-{c[2]}x{c[3]}" for c in CASES])
def test_noalloc_matches_zo_perturb_on_two_calls(lib, gpu, dtype, r, m, n):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    seed, base, eps = 8080, 17, 1e-1
    W0 = make_weight(m, n, dtype, 5, gpu)
    z = SubZeroPlus([W0.clone()], r, 4, seed, matrix_index_base=base)
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, 1)   # the fp32-FMA arithmetic of the variant
    z.init_subspace(0)
    torch.cuda.synchronize()
    U, V = to_f64(z.U[0]), to_f64(z.V[0])
    W = W0.clone()
    for t, qa, ca, qb, cb in [(0, 0, 1.0, -1, 0.0), (0, 0, -2.0, 1, 1.0)]:
        before = to_f64(W)
        z.perturb(t, qa, ca, qb, cb, eps)
        zb.zo_perturb_noalloc(W, z.U[0], z.V[0], r, seed, base, t, qa, ca, qb, cb, eps)
        torch.cuda.synchronize()
        # the same kernels on the same inputs: bit for bit the context's result
        assert torch.equal(W, z.weights[0]), f"no-alloc t={t} qa={qa} differs from zo_perturb"
        # and the oracle's pass within 1 ulp (bf16) / rel 1e-5 (fp32) at the operand scale
        terms = [(qa, ca)] + ([(qb, cb)] if qb >= 0 else [])
        C = subzero.perturb_coeff(seed, base, t, r, terms, f32(eps))
        want = subzero.apply_pass(before, dtype, U, V, C)
        zc = abs(f32(eps)) * sum(abs(c) for _, c in terms)
        assert_weights(to_f64(W), want, dtype, f"no-alloc t={t} qa={qa} vs oracle", before=before,
                       terms=update_terms(U, C, V, zc))
    assert not torch.equal(W, W0)                         # the passes did change W
    z.sync()
    z.close()


def test_noalloc_leaves_free_device_memory_unchanged(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    m, n, r = 512, 2048, 32
    W = make_weight(m, n, "bf16", 6, gpu)
    U = torch.linalg.qr(torch.randn(m, r, device=gpu))[0].contiguous()
    V = torch.linalg.qr(torch.randn(n, r, device=gpu))[0].contiguous()
    zb.zo_perturb_noalloc(W, U, V, r, 3, 0, 0, 0, 1.0, -1, 0.0, 1e-3)   # first call: set-up
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for k in range(3):
        zb.zo_perturb_noalloc(W, U, V, r, 3, 0, 0, k % 4, 1.0, -1, 0.0, 1e-3)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"device free memory moved by {free0 - free1} bytes"


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

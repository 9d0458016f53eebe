"""Failure detection on the GPU without a GPU fault.

Every mbarrier wait of the tensor-core weight passes is bounded (both kernels: r <= 32
with the operands in shared memory, r >= 64 with U in Tensor Memory).  The test hook
ZO_OPTION_TEST_WAIT_TIMEOUT makes one CTA of the next pass wait on a barrier that
nothing arrives on (a flag nothing sets); its wait runs out after ~0.1 s, the kernel
records a timeout in the context's status word, the other roles of that CTA stop
and release what they hold, and every other CTA finishes normally.  The host must
see ZO_ERR_TIMEOUT, and the context must keep working afterwards."""

import pytest

from gpu_util import make_weight, oracle_perturb, snapshot
from parity import assert_weights

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("r", [32, 64, 128])
def test_expired_wait_reports_timeout_and_the_context_recovers(lib, gpu, r):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    base, seed = 40, 6060
    z = SubZeroPlus([make_weight(300, 520, "bf16", 1, gpu), make_weight(1030, 264, "bf16", 2, gpu)],
                    r, 2, seed, matrix_index_base=base)
    z.init_subspace(0)
    z.perturb(0, 0, 1.0, -1, 0.0, 1e-3)
    z.sync()
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TEST_WAIT_TIMEOUT, 1)
    z.perturb(0, 0, -1.0, -1, 0.0, 1e-3)
    assert zb.zo_wpass_path(z.ctx) == 2
    with pytest.raises(zb.ZoError) as e:
        z.sync()
    assert e.value.status == zb.ZO_ERR_TIMEOUT
    # the status word was cleared and the hook was one-shot: the next pass is normal
    z.sync()
    before = snapshot(z)
    z.perturb(1, 1, 1.0, -1, 0.0, 1e-1)
    after = snapshot(z)
    z.sync()
    for i in range(2):
        want, T = oracle_perturb(before, i, "bf16", seed, base + i, 1, r, [(1, 1.0)], 1e-1)
        assert_weights(after["W"][i], want, "bf16", f"after recovery, matrix {i}",
                       before=before["W"][i], terms=T)
    z.close()


def test_linear_pair_wait_reports_timeout_and_the_context_recovers(lib, gpu):
    """The SM-pair perturbed-linear launch: with the hook armed its Y tiles wait for S rows
    that are never counted as written (the row-block counters' epoch is one ahead); every
    such wait gives up after ~0.1 s, the launch reports a timeout, zo_sync_status zeroes the
    counters, and the next call is exact again."""
    import torch
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    from oracle import subzero
    from gpu_util import f32
    from test_gpu_linear import _check, _tokens
    base, seed = 50, 7070
    z = SubZeroPlus([make_weight(304, 520, "bf16", 4, gpu)], 32, 2, seed, matrix_index_base=base)
    z.init_subspace(0)
    zb.zo_linear_prepare(z.ctx, 3, 0, 1.0, 1, -1.0, 1e-2)
    X = _tokens(700, 520, 12, gpu)
    Y = torch.empty((700, 304), dtype=torch.bfloat16, device=gpu)
    zb.zo_linear_perturbed(z.ctx, 0, X, Y)          # a normal call first: counters in use
    z.sync()
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TEST_WAIT_TIMEOUT, 1)
    zb.zo_linear_perturbed(z.ctx, 0, X, Y)
    assert zb.zo_linear_tiling(z.ctx) >= 4
    with pytest.raises(zb.ZoError) as e:
        z.sync()
    assert e.value.status == zb.ZO_ERR_TIMEOUT
    z.sync()                                         # cleared; the hook was one-shot
    before = snapshot(z)
    Y.fill_(float("nan"))
    zb.zo_linear_perturbed(z.ctx, 0, X, Y)
    z.sync()
    C = subzero.perturb_coeff(seed, base, 3, 32, [(0, 1.0), (1, -1.0)], f32(1e-2))
    _check(Y, X, before["W"][0], before["U"][0], before["V"][0], C, 2.0 * f32(1e-2),
           "perturbed linear after the expired wait")
    z.close()


def test_wait_hook_needs_the_tensor_core_pass(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    z = SubZeroPlus([make_weight(64, 64, "f32", 3, gpu)], 8, 2, 1)
    with pytest.raises(zb.ZoError) as e:
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_TEST_WAIT_TIMEOUT, 1)
    assert e.value.status == zb.ZO_ERR_UNSUPPORTED
    z.close()


def test_rejected_tensor_core_descriptor_is_refused_not_downgraded(lib, gpu):
    # A bf16 set at r = 16 qualifies for the tensor-core pass.  A W row stride of 2^40
    # bytes is one cuTensorMapEncodeTiled rejects (strides must stay below 2^40), so the
    # context cannot build that pass.  zo_create still succeeds, but the automatic path
    # refuses zo_perturb / zo_step with ZO_ERR_UNSUPPORTED (naming the remedy) instead of
    # running the FMA pass in its place, and nothing is launched.  The context is only
    # created and destroyed: no kernel ever touches this W.
    import torch
    from paper_2608_15665_gb300 import binding as zb
    m, n, r = 16, 64, 16
    W = torch.zeros(m, n, dtype=torch.bfloat16, device=gpu)
    bufs = [torch.zeros(m, r, device=gpu), torch.zeros(n, r, device=gpu),
            torch.zeros(r, r, device=gpu), torch.zeros(r, r, device=gpu)]
    mat = zb.zo_matrix(W.data_ptr(), m, n, 2 ** 39, zb.ZO_BF16, 0, *[b.data_ptr() for b in bufs])
    ctx = zb.zo_create([mat], r, 2, 1)
    try:
        with pytest.raises(zb.ZoError) as e:
            zb.zo_perturb(ctx, 0, 0, 1.0, -1, 0.0, 1e-3)
        assert e.value.status == zb.ZO_ERR_UNSUPPORTED
        assert "ZO_OPTION_WPASS_PATH" in str(e.value) and "W_0" in str(e.value)
        losses = torch.full((4,), 2.0, device=gpu)
        with pytest.raises(zb.ZoError) as e:
            zb.zo_step(ctx, 0, 1, losses, zb.ZO_SCHEME_CENTRAL, 1e-3, 1e-3, 0.9, 0.95, 1e-8, 1, 1.0)
        assert e.value.status == zb.ZO_ERR_UNSUPPORTED
        assert zb.zo_kernel_launches(ctx) == 0
        # the tensor-core path cannot be forced either
        with pytest.raises(zb.ZoError) as e:
            zb.zo_set_option(ctx, zb.ZO_OPTION_WPASS_PATH, 2)
        assert e.value.status == zb.ZO_ERR_UNSUPPORTED
    finally:
        zb.zo_destroy(ctx)

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


def test_wait_hook_needs_the_tensor_core_pass(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    z = SubZeroPlus([make_weight(64, 64, "f32", 3, gpu)], 8, 2, 1)
    with pytest.raises(zb.ZoError) as e:
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_TEST_WAIT_TIMEOUT, 1)
    assert e.value.status == zb.ZO_ERR_UNSUPPORTED
    z.close()
